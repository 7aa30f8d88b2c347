"""Python binding of libmoeca.so (include/moeca.h): ctypes marshalling only.

The functions keep the C names (moeca_create, moeca_step, ...) and raise
MoecaError on a non-OK status.  Every step of the layer runs in the CUDA
library; there is no Python or CPU fallback: importing this module fails
loudly when the library has not been built.  ``Stack`` is a convenience
wrapper that holds torch tensors (device memory) and passes their pointers.
"""
from __future__ import annotations

import ctypes as C
import math
import os
import re

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libmoeca.so")
INCLUDE = os.path.join(os.path.dirname(PKG), "include")
HEADER = os.path.join(INCLUDE, "moeca.h")

MOECA_OK = 0
MOECA_ERR_INVALID_ARG, MOECA_ERR_UNSUPPORTED, MOECA_ERR_CUDA, MOECA_ERR_OOM = -1, -2, -3, -4
MOECA_ERR_STATE, MOECA_ERR_TIMEOUT, MOECA_ERR_DEVICE_STATUS = -5, -6, -7
STATUS_NAMES = {0: "OK", -1: "INVALID_ARG", -2: "UNSUPPORTED", -3: "CUDA", -4: "OOM", -5: "STATE",
                -6: "TIMEOUT", -7: "DEVICE_STATUS"}
MOECA_F32, MOECA_BF16 = 0, 1
MOECA_FFN_AUTO, MOECA_FFN_SIMT = 0, 1
KERNEL_KINDS = ["router", "select", "compact", "ffn1", "ffn2", "combine", "prep", "ffn",
                "qkv", "attn", "oproj", "attn_aux", "adaln"]
ATTN_SYNC, ATTN_STALE, ATTN_FULL = 0, 1, 2


class moeca_config(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("hidden", C.c_int32), ("ffn", C.c_int32),
                ("n_experts", C.c_int32), ("top_k", C.c_int32), ("n_shared", C.c_int32),
                ("max_tokens", C.c_int32), ("dtype", C.c_int32),
                ("lambda1", C.c_float), ("lambda2", C.c_float), ("tau0", C.c_float),
                ("alpha", C.c_float), ("beta", C.c_float),
                ("refresh_period", C.c_int32), ("renorm_topk", C.c_int32), ("entropy_norm", C.c_int32),
                ("shared_policy", C.c_int32), ("reused_meta_policy", C.c_int32),
                ("gelu_tanh", C.c_int32), ("ffn_impl", C.c_int32), ("ffn_tile_n", C.c_int32),
                ("ffn_split_k", C.c_int32), ("score_terms", C.c_int32), ("granularity", C.c_int32),
                ("n_heads", C.c_int32), ("seq_len", C.c_int32), ("attn_policy", C.c_int32),
                ("attn_impl", C.c_int32), ("adaln", C.c_int32), ("ln_eps", C.c_float),
                ("keep_route_in", C.c_int32), ("token_reuse_policy", C.c_int32), ("combine_direct", C.c_int32),
                ("weight_prefetch_mb", C.c_int32)]


class moeca_layer_weights(C.Structure):
    _fields_ = [("w_gate", C.c_void_p), ("b_gate", C.c_void_p), ("w1", C.c_void_p),
                ("w2", C.c_void_p), ("ws1", C.c_void_p), ("ws2", C.c_void_p),
                ("w_qkv", C.c_void_p), ("b_qkv", C.c_void_p), ("w_o", C.c_void_p), ("b_o", C.c_void_p),
                ("w_ada", C.c_void_p), ("b_ada", C.c_void_p)]


class moeca_step_args(C.Structure):
    _fields_ = [("n_tokens", C.c_int32), ("step_index", C.c_int32), ("force_refresh", C.c_int32),
                ("tau0_override", C.c_float), ("cond", C.c_void_p)]


class moeca_stats(C.Structure):
    _fields_ = [(n, C.c_int64) for n in (
        "layer_steps", "refresh_layer_steps", "branches", "cache_step_branches", "matched",
        "recomputed", "reused", "tokens_fully_reused", "shared_recomputed",
        "near_margin_route", "near_margin_score")] + [("device_status", C.c_int32),
                                                      ("device_detail", C.c_int32),
                                                      ("attn_recomputed", C.c_int64)]

    def as_dict(self) -> dict:
        return {n: getattr(self, n) for n, _ in self._fields_}


class moeca_layer_state(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("cache_e", "cache_w", "cache_norm", "cache_h", "shared_h", "ema",
                                            "attn_a", "cache_y")]


class moeca_layer_trace(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("route_e", "route_w", "tau", "recompute", "slot", "matched",
                                            "token_any", "counts", "offsets", "list", "layer_in",
                                            "block_in", "route_in", "resid", "mod")]


class moeca_shard(C.Structure):
    _fields_ = [("rank", C.c_int32), ("world", C.c_int32), ("total_tokens", C.c_int32)]


class moeca_kernel_times(C.Structure):
    _fields_ = [("total_ms", C.c_double * 13), ("launches", C.c_int64 * 13)]


class moeca_route_args(C.Structure):
    _fields_ = [("dtype", C.c_int32), ("n_tokens", C.c_int32), ("hidden", C.c_int32),
                ("n_experts", C.c_int32), ("top_k", C.c_int32), ("renorm_topk", C.c_int32),
                ("entropy_norm", C.c_int32), ("beta", C.c_float), ("tau0", C.c_float), ("alpha", C.c_float),
                ("x", C.c_void_p), ("w_gate", C.c_void_p), ("b_gate", C.c_void_p), ("ema", C.c_void_p),
                ("route_e", C.c_void_p), ("route_w", C.c_void_p), ("tau", C.c_void_p)]


class moeca_ddpm_args(C.Structure):
    _fields_ = [("n", C.c_int64), ("eps_dtype", C.c_int32), ("alpha", C.c_double), ("alpha_bar", C.c_double),
                ("sigma", C.c_double), ("x_t", C.c_void_p), ("eps", C.c_void_p), ("z", C.c_void_p),
                ("x_prev", C.c_void_p), ("x_next", C.c_void_p)]


class MoecaError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with paper_2606_15615_gb300.build.build()")
    lib = C.CDLL(LIB_PATH)
    H = C.c_void_p
    sig = {
        "moeca_config_default": (None, [C.POINTER(moeca_config)]),
        "moeca_create": (C.c_int, [C.POINTER(moeca_config), C.POINTER(moeca_layer_weights), C.c_int32,
                                   C.POINTER(H)]),
        "moeca_step": (C.c_int, [H, C.c_void_p, C.c_void_p, C.POINTER(moeca_step_args), C.c_void_p]),
        "moeca_step_host": (C.c_int, [H, C.c_void_p, C.c_void_p, C.POINTER(moeca_step_args), C.c_void_p]),
        "moeca_host_join": (C.c_int, [H, C.c_void_p]),
        "moeca_shard_exchange_bytes": (C.c_int, [H, C.c_int32, C.POINTER(C.c_int64)]),
        "moeca_shard_begin": (C.c_int, [H, C.c_void_p, C.c_void_p, C.POINTER(moeca_step_args),
                                        C.POINTER(moeca_shard), C.c_void_p, C.c_void_p, C.c_void_p]),
        "moeca_shard_next": (C.c_int, [H, C.c_void_p, C.POINTER(C.c_int32)]),
        "moeca_get_stats": (C.c_int, [H, C.c_int32, C.POINTER(moeca_stats)]),
        "moeca_reset_stats": (C.c_int, [H]),
        "moeca_get_layer_state": (C.c_int, [H, C.c_int32, C.POINTER(moeca_layer_state),
                                            C.POINTER(C.c_int32), C.c_void_p]),
        "moeca_set_layer_state": (C.c_int, [H, C.c_int32, C.POINTER(moeca_layer_state), C.c_int32,
                                            C.c_void_p]),
        "moeca_get_layer_trace": (C.c_int, [H, C.c_int32, C.POINTER(moeca_layer_trace), C.c_void_p]),
        "moeca_reset": (C.c_int, [H]),
        "moeca_inject_fault": (C.c_int, [H, C.c_int32]),
        "moeca_set_kernel_timing": (C.c_int, [H, C.c_int32]),
        "moeca_get_kernel_times": (C.c_int, [H, C.POINTER(moeca_kernel_times), C.c_int32]),
        "moeca_destroy": (C.c_int, [H]),
        "moeca_status_string": (C.c_char_p, [C.c_int]),
        "moeca_last_error": (C.c_char_p, [H]),
        "moeca_route_noalloc": (C.c_int, [C.POINTER(moeca_route_args), C.c_void_p]),
        "moeca_ddpm_schedule": (C.c_int, [C.c_int32, C.c_int32, C.c_double, C.c_double, C.POINTER(C.c_int32),
                                          C.POINTER(C.c_double), C.POINTER(C.c_double), C.POINTER(C.c_double)]),
        "moeca_ddpm_step": (C.c_int, [C.POINTER(moeca_ddpm_args), C.c_void_p]),
        "moeca_probe_ffma": (C.c_int32, [C.c_int32, C.c_int32, C.POINTER(C.c_double), C.POINTER(C.c_double)]),
        "moeca_probe_stream": (C.c_int32, [C.c_int32, C.c_int64, C.c_int32, C.c_int32, C.c_int32,
                                           C.POINTER(C.c_double), C.POINTER(C.c_double)]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


LIB = _load()


def header_functions() -> list:
    """Names of the functions the headers under include/ declare."""
    names = set()
    for fn in sorted(os.listdir(INCLUDE)):
        if fn.endswith(".h"):
            with open(os.path.join(INCLUDE, fn)) as f:
                text = re.sub(r"/\*.*?\*/", "", f.read(), flags=re.S)
            names |= set(re.findall(r"\b(moeca_[a-z_]+)\s*\(", text))
    return sorted(names)


def _check(status: int, handle=None):
    if status != MOECA_OK:
        msg = LIB.moeca_last_error(handle)
        raise MoecaError(status, msg.decode() if msg else "")


def moeca_config_default(**kw) -> moeca_config:
    cfg = moeca_config()
    LIB.moeca_config_default(C.byref(cfg))
    for k, v in kw.items():
        if not hasattr(cfg, k):
            raise AttributeError(k)
        setattr(cfg, k, v)
    return cfg


def moeca_create(cfg: moeca_config, layers: list, device: int = 0):
    arr = (moeca_layer_weights * len(layers))(*layers)
    h = C.c_void_p()
    _check(LIB.moeca_create(C.byref(cfg), arr, device, C.byref(h)))
    return h


def moeca_step(h, x_in_ptr: int, x_out_ptr: int, n_tokens: int, step_index: int,
               force_refresh: bool = False, tau0_override: float = math.nan, stream: int = 0,
               cond_ptr: int | None = None):
    args = moeca_step_args(n_tokens, step_index, int(force_refresh), tau0_override, cond_ptr)
    _check(LIB.moeca_step(h, x_in_ptr, x_out_ptr, C.byref(args), stream or None), h)


def moeca_step_host(h, x_in_host_ptr: int, x_out_host_ptr: int, n_tokens: int, step_index: int,
                    force_refresh: bool = False, tau0_override: float = math.nan, stream: int = 0,
                    cond_host_ptr: int | None = None):
    """One step from and to host buffers (see include/moeca.h); asynchronous."""
    args = moeca_step_args(n_tokens, step_index, int(force_refresh), tau0_override, cond_host_ptr)
    _check(LIB.moeca_step_host(h, x_in_host_ptr, x_out_host_ptr, C.byref(args), stream or None), h)


def moeca_host_join(h, stream: int = 0):
    """Order ``stream`` after every upload and read-back of moeca_step_host."""
    _check(LIB.moeca_host_join(h, stream or None), h)


def moeca_shard_exchange_bytes(h, n_tokens: int) -> int:
    """Bytes one rank contributes to each layer's exchange (see include/moeca.h)."""
    n = C.c_int64()
    _check(LIB.moeca_shard_exchange_bytes(h, n_tokens, C.byref(n)), h)
    return n.value


def moeca_shard_begin(h, x_in_ptr: int, x_out_ptr: int, n_tokens: int, step_index: int, rank: int, world: int,
                      send_ptr: int, recv_ptr: int, force_refresh: bool = False, tau0_override: float = math.nan,
                      stream: int = 0):
    args = moeca_step_args(n_tokens, step_index, int(force_refresh), tau0_override, None)
    sh = moeca_shard(rank, world, world * n_tokens)
    _check(LIB.moeca_shard_begin(h, x_in_ptr, x_out_ptr, C.byref(args), C.byref(sh), send_ptr, recv_ptr,
                                 stream or None), h)


def moeca_shard_next(h, stream: int = 0) -> bool:
    done = C.c_int32()
    _check(LIB.moeca_shard_next(h, stream or None, C.byref(done)), h)
    return bool(done.value)


def torch_allgather(group=None):
    """The exchange of a token-sharded step over torch.distributed: every
    rank's send bytes into recv in rank order (NCCL on the current stream)."""
    import torch.distributed as dist

    def exchange(send, recv):
        if dist.get_backend(group) == "nccl":
            dist.all_gather_into_tensor(recv, send, group=group)
        else:  # gloo: the list form, into views of recv in rank order
            dist.all_gather(list(recv.chunk(dist.get_world_size(group))), send, group=group)
    return exchange


def moeca_get_stats(h, layer: int = -1) -> dict:
    st = moeca_stats()
    _check(LIB.moeca_get_stats(h, layer, C.byref(st)), h)
    return st.as_dict()


def moeca_reset_stats(h):
    _check(LIB.moeca_reset_stats(h), h)


def moeca_get_layer_state(h, layer: int, dst: moeca_layer_state, stream: int = 0) -> int:
    n = C.c_int32()
    _check(LIB.moeca_get_layer_state(h, layer, C.byref(dst), C.byref(n), stream or None), h)
    return n.value


def moeca_set_layer_state(h, layer: int, src: moeca_layer_state, n_tokens: int, stream: int = 0):
    _check(LIB.moeca_set_layer_state(h, layer, C.byref(src), n_tokens, stream or None), h)


def moeca_get_layer_trace(h, layer: int, dst: moeca_layer_trace, stream: int = 0):
    _check(LIB.moeca_get_layer_trace(h, layer, C.byref(dst), stream or None), h)


def moeca_reset(h):
    _check(LIB.moeca_reset(h), h)


MOECA_FAULT_BARRIER_STALL = 1


def moeca_inject_fault(h, kind: int):
    """Test hook: arm a host-side fault for the next step (see include/moeca.h)."""
    _check(LIB.moeca_inject_fault(h, kind), h)


def moeca_set_kernel_timing(h, enable: bool):
    _check(LIB.moeca_set_kernel_timing(h, int(enable)), h)


def moeca_get_kernel_times(h, reset: bool = False) -> dict:
    kt = moeca_kernel_times()
    _check(LIB.moeca_get_kernel_times(h, C.byref(kt), int(reset)), h)
    return {n: (kt.total_ms[i], kt.launches[i]) for i, n in enumerate(KERNEL_KINDS)}


def moeca_destroy(h):
    if h is not None and h.value:
        _check(LIB.moeca_destroy(h))


def moeca_route_noalloc(args: moeca_route_args, stream: int = 0):
    """The allocation-free router of one layer (see include/moeca.h)."""
    st = LIB.moeca_route_noalloc(C.byref(args), stream or None)
    if st != MOECA_OK:
        raise MoecaError(st, "moeca_route_noalloc")


def moeca_ddpm_schedule(n_steps: int, n_train: int = 1000, beta_start: float = 1e-4, beta_end: float = 0.02):
    """Per-step (t, alpha, alpha_bar, beta) lists of a sampling run (Eq. 1; see include/moeca.h)."""
    t = (C.c_int32 * n_steps)()
    al, ab, be = (C.c_double * n_steps)(), (C.c_double * n_steps)(), (C.c_double * n_steps)()
    st = LIB.moeca_ddpm_schedule(n_steps, n_train, beta_start, beta_end, t, al, ab, be)
    if st != MOECA_OK:
        _check(st, None)
    return list(t), list(al), list(ab), list(be)


def moeca_ddpm_step(args: moeca_ddpm_args, stream: int = 0):
    """One reverse transition of Eq. 1 on device buffers (see include/moeca.h)."""
    st = LIB.moeca_ddpm_step(C.byref(args), stream or None)
    if st != MOECA_OK:
        _check(st, None)


def moeca_probe_ffma(device: int = 0, iterations: int = 1 << 16) -> tuple:
    """Measured fp32 FFMA throughput of ``device``: (TFLOP/s, ms) (include/moeca_probe.h)."""
    tf, ms = C.c_double(), C.c_double()
    st = LIB.moeca_probe_ffma(device, iterations, C.byref(tf), C.byref(ms))
    if st != 0:
        raise MoecaError(st, "moeca_probe_ffma")
    return tf.value, ms.value


def moeca_probe_stream(device: int, n_tokens: int, rows: int, row_bytes: int, reps: int = 15) -> tuple:
    """Streaming rate of ``device`` at one shape: (GB/s, median us) of a kernel
    that reads ``rows`` rows of ``row_bytes`` per token and writes one
    (include/moeca_probe.h)."""
    gbs, us = C.c_double(), C.c_double()
    st = LIB.moeca_probe_stream(device, n_tokens, rows, row_bytes, reps, C.byref(gbs), C.byref(us))
    if st != 0:
        raise MoecaError(st, "moeca_probe_stream")
    return gbs.value, us.value


def moeca_status_string(status: int) -> str:
    return LIB.moeca_status_string(status).decode()


# ---------------------------------------------------------------------------
# torch convenience wrapper (device memory + streams only)
# ---------------------------------------------------------------------------

class Stack:
    """A MoECa layer stack on one GPU, fed with torch CUDA tensors.

    ``layer_weights`` is a list of dicts of numpy float32 arrays (bf16-exact
    for bf16) as made by ``workloads.make_layer_weights``; they are copied to
    the device once and kept alive here.
    """

    def __init__(self, cfg: moeca_config, layer_weights: list, device: int = 0):
        import numpy as np
        import torch
        self.torch = torch
        self.cfg = cfg
        self.device = torch.device("cuda", device)
        self.dtype = torch.bfloat16 if cfg.dtype == MOECA_BF16 else torch.float32
        self._keep = []
        cl = []
        for w in layer_weights:
            def dev(a, dt=self.dtype):
                if a is None:
                    return None
                if isinstance(a, torch.Tensor):
                    t = a.to(self.device).to(dt).contiguous()
                else:
                    t = torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(self.device).to(dt).contiguous()
                self._keep.append(t)
                return t
            lw = moeca_layer_weights()
            lw.w_gate = dev(w["w_gate"]).data_ptr()
            b = dev(w.get("b_gate"), torch.float32)
            lw.b_gate = b.data_ptr() if b is not None else None
            lw.w1 = dev(w["w1"]).data_ptr()
            lw.w2 = dev(w["w2"]).data_ptr()
            if cfg.n_shared:
                lw.ws1 = dev(w["ws1"][0]).data_ptr()
                lw.ws2 = dev(w["ws2"][0]).data_ptr()
            if cfg.n_heads:
                lw.w_qkv = dev(w["w_qkv"]).data_ptr()
                lw.w_o = dev(w["w_o"]).data_ptr()
                for name in ("b_qkv", "b_o"):
                    bt = dev(w.get(name), torch.float32)
                    setattr(lw, name, bt.data_ptr() if bt is not None else None)
            if cfg.adaln:
                lw.w_ada = dev(w["w_ada"]).data_ptr()
                bt = dev(w.get("b_ada"), torch.float32)
                lw.b_ada = bt.data_ptr() if bt is not None else None
            cl.append(lw)
        self.handle = moeca_create(cfg, cl, device)

    def close(self):
        if getattr(self, "handle", None) is not None:
            moeca_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def stream_ptr(self) -> int:
        return self.torch.cuda.current_stream(self.device).cuda_stream

    def step(self, x, step_index: int, force_refresh: bool = False, tau0=math.nan, out=None, cond=None):
        """One denoising step; ``cond`` is the [T / seq_len, D] float32 CUDA
        tensor of per-sample conditioning an AdaLN stack reads."""
        torch = self.torch
        T = x.shape[0]
        if out is None:
            out = torch.empty_like(x)
        if cond is not None:
            if cond.dtype != torch.float32 or not cond.is_cuda or not cond.is_contiguous():
                raise ValueError("cond must be a contiguous float32 CUDA tensor")
            samples = T // (self.cfg.seq_len or T) if T else 0
            if cond.numel() != samples * self.cfg.hidden:
                raise ValueError(f"cond must hold {samples} x {self.cfg.hidden} values (one row per sample)")
            self._cond = cond  # read by the step's first kernel: keep it alive until then
        moeca_step(self.handle, x.data_ptr(), out.data_ptr(), T, step_index, force_refresh, tau0,
                   self.stream_ptr(), cond.data_ptr() if cond is not None else None)
        return out

    def step_sharded(self, x, step_index: int, rank: int, world: int, exchange, force_refresh: bool = False,
                     tau0=math.nan, out=None):
        """One denoising step of this rank's slice ``x`` [n_tokens, D] of a
        token-sharded batch (include/moeca.h): each layer's entropy partials
        are exchanged with ``exchange(send, recv)`` (uint8 CUDA tensors:
        ``send`` this rank's bytes, ``recv`` world x that, filled in rank
        order), e.g. ``torch_allgather()``."""
        torch = self.torch
        T = x.shape[0]
        if out is None:
            out = torch.empty_like(x)
        nbytes = moeca_shard_exchange_bytes(self.handle, T)
        if getattr(self, "_xbuf", None) is None or self._xbuf[0].numel() < nbytes or \
                self._xbuf[1].numel() < world * nbytes:
            self._xbuf = (self._empty((nbytes,), torch.uint8), self._empty((world * nbytes,), torch.uint8))
        send, recv = self._xbuf[0][:nbytes], self._xbuf[1][:world * nbytes]
        sp = self.stream_ptr()
        moeca_shard_begin(self.handle, x.data_ptr(), out.data_ptr(), T, step_index, rank, world, send.data_ptr(),
                          recv.data_ptr(), force_refresh, tau0, sp)
        while True:
            exchange(send, recv)
            if moeca_shard_next(self.handle, sp):
                return out

    def _empty(self, shape, dtype):
        return self.torch.empty(shape, dtype=dtype, device=self.device)

    def get_state(self, layer: int) -> dict:
        torch = self.torch
        c = self.cfg
        T = c.max_tokens
        t = dict(cache_e=self._empty((T, c.top_k), torch.int32), cache_w=self._empty((T, c.top_k), torch.float32),
                 cache_norm=self._empty((T, c.top_k), torch.float32),
                 cache_h=self._empty((T, c.top_k, c.hidden), self.dtype),
                 shared_h=self._empty((T, c.hidden), self.dtype) if c.n_shared else None,
                 ema=self._empty((T, c.n_experts), torch.float32),
                 attn_a=self._empty((T, c.hidden), self.dtype) if c.n_heads else None,
                 cache_y=self._empty((T, c.hidden), torch.float32) if c.token_reuse_policy else None)
        st = moeca_layer_state(**{k: (v.data_ptr() if v is not None else None) for k, v in t.items()})
        n = moeca_get_layer_state(self.handle, layer, st, self.stream_ptr())
        return {k: (v[:n] if v is not None else None) for k, v in t.items()} | {"n_tokens": n}

    def set_state(self, layer: int, state: dict):
        n = int(state["cache_e"].shape[0])
        keep = {k: v.contiguous() for k, v in state.items() if k != "n_tokens" and v is not None}
        st = moeca_layer_state(**{k: keep[k].data_ptr() if k in keep else None
                                  for k in ("cache_e", "cache_w", "cache_norm", "cache_h", "shared_h", "ema",
                                            "attn_a", "cache_y")})
        moeca_set_layer_state(self.handle, layer, st, n, self.stream_ptr())
        self.torch.cuda.current_stream(self.device).synchronize()

    def get_trace(self, layer: int, n_tokens: int) -> dict:
        torch = self.torch
        c = self.cfg
        T, k, G = n_tokens, c.top_k, c.n_experts + c.n_shared
        t = dict(route_e=self._empty((T, k), torch.int32), route_w=self._empty((T, k), torch.float32),
                 tau=self._empty((c.n_experts,), torch.float32), recompute=self._empty((T, k), torch.uint8),
                 slot=self._empty((T, k), torch.int8), matched=self._empty((T, k), torch.uint8),
                 token_any=self._empty((T,), torch.uint8), counts=self._empty((G,), torch.int32),
                 offsets=self._empty((G + 1,), torch.int32),
                 list=self._empty((T * (k + c.n_shared),), torch.int32),
                 layer_in=self._empty((T, c.hidden), self.dtype),
                 block_in=self._empty((T, c.hidden), self.dtype) if c.n_heads else None,
                 route_in=self._empty((T, c.hidden), self.dtype) if c.adaln and c.keep_route_in else None,
                 resid=self._empty((T, c.hidden), self.dtype) if c.n_heads else None,
                 mod=self._empty((T // (c.seq_len or T), 6 * c.hidden), torch.float32) if c.adaln else None)
        t = {kk: v for kk, v in t.items() if v is not None}
        tr = moeca_layer_trace(**{kk: v.data_ptr() for kk, v in t.items()})
        moeca_get_layer_trace(self.handle, layer, tr, self.stream_ptr())
        return t

    def stats(self, layer: int = -1) -> dict:
        return moeca_get_stats(self.handle, layer)


def ddpm_step(x_t, eps, alpha: float, alpha_bar: float, sigma: float, z=None, x_prev=None, x_next=None,
              stream: int = 0):
    """Eq. 1 on torch CUDA tensors: x_prev (fp32) = the reverse step of x_t
    (fp32) with the denoiser output eps; x_next (eps's dtype) optionally
    receives x_prev for the next denoiser call.  Returns x_prev."""
    import torch
    if x_prev is None:
        x_prev = torch.empty_like(x_t)
    args = moeca_ddpm_args(
        x_t.numel(), MOECA_BF16 if eps.dtype == torch.bfloat16 else MOECA_F32, alpha, alpha_bar, sigma,
        x_t.data_ptr(), eps.data_ptr(), z.data_ptr() if z is not None else None, x_prev.data_ptr(),
        x_next.data_ptr() if x_next is not None else None)
    moeca_ddpm_step(args, stream or torch.cuda.current_stream(x_t.device).cuda_stream)
    return x_prev
