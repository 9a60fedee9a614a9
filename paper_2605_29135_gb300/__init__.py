"""GB300-native capped-residency MoE decode step (Python binding of libmoe.so).

The paper's residency problem (Section "Rotary GPU Concept", Fig. 1): expert weights live in a
pinned host tier, a fixed group of GPU slots holds a subset of them, a lookup table maps
expert id -> slot, and the routing result drives selective loads and evictions. One decode step
runs the router / top-k, the slot lookup with deterministic LRU eviction (lower id on ties), the
miss copies on a side stream, the SwiGLU expert GEMVs and the rank-ordered combine, all inside
libmoe.so. This module only marshals arguments; the method names follow the C ABI
(include/moe.h) without the ``moe_`` prefix.
"""
from __future__ import annotations

import ctypes

import numpy as np

from . import _lib
from ._lib import (BATCHED_PATH, DTYPE, POLICY, SCHEDULE, STATUS, DecoderConfig, KernelTime, MoeConfig, Stats,
                   TraceRec)

TRACE_DTYPE = np.dtype([("step", np.int32), ("layer", np.int32), ("expert", np.int32), ("kind", np.int32),
                        ("slot", np.int32), ("evicted", np.int32)])


class MoEError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


def make_config(d, n_experts, top_k, d_ff, n_layers, wdtype, adtype, cap_slots=0, cap_bytes=0, renorm=True,
                device=0, max_batch=1, trace_capacity=1 << 22, device_pool=None, schedule="device",
                miss_ctas=0, batched_path="auto", policy="lru", lookahead=False) -> MoeConfig:
    return MoeConfig(d=d, n_experts=n_experts, top_k=top_k, d_ff=d_ff, n_layers=n_layers, max_batch=max_batch,
                     wdtype=DTYPE[wdtype], adtype=DTYPE[adtype], cap_slots=cap_slots, cap_bytes=cap_bytes,
                     renorm=1 if renorm else 0, device=device, device_pool=device_pool,
                     trace_capacity=trace_capacity, schedule=SCHEDULE[schedule], miss_ctas=miss_ctas,
                     batched_path=BATCHED_PATH[batched_path], policy=POLICY[policy],
                     lookahead=1 if lookahead else 0)


def expert_bytes(cfg: MoeConfig) -> int:
    return int(_lib.load().moe_expert_bytes(ctypes.byref(cfg)))


def pool_bytes(cfg: MoeConfig) -> int:
    return int(_lib.load().moe_pool_bytes(ctypes.byref(cfg)))


def _ptr(a) -> ctypes.c_void_p:
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        if not a.flags["C_CONTIGUOUS"]:
            raise ValueError("arrays passed to libmoe must be C-contiguous")
        return ctypes.c_void_p(a.ctypes.data)
    # torch tensor
    if not a.is_contiguous():
        raise ValueError("tensors passed to libmoe must be contiguous")
    return ctypes.c_void_p(a.data_ptr())


def _nbytes(a) -> int:
    return a.nbytes if isinstance(a, np.ndarray) else a.numel() * a.element_size()


def _check_buffer(name: str, a, need: int, where: str, device: int = 0):
    """Refuse a buffer the library would read or write past its end, or on the wrong side."""
    if a is None:
        raise ValueError(f"{name} is None")
    if not (a.flags["C_CONTIGUOUS"] if isinstance(a, np.ndarray) else a.is_contiguous()):
        raise ValueError(f"{name} must be contiguous")
    on_gpu = not isinstance(a, np.ndarray) and a.is_cuda
    if where == "device" and (not on_gpu or a.device.index != device):
        raise ValueError(f"{name} must be a tensor on cuda:{device}")
    if where == "host" and on_gpu:
        raise ValueError(f"{name} must be in host memory")
    if _nbytes(a) < need:
        raise ValueError(f"{name} holds {_nbytes(a)} bytes, the call needs {need}")


def _weight_bytes(wdtype: int, n: int) -> int:
    """Bytes of n stored weight elements (int4: two per byte)."""
    return {DTYPE["fp32"]: 4 * n, DTYPE["bf16"]: 2 * n, DTYPE["int4"]: n // 2}[wdtype]


class MoE:
    """One library handle (moe_create ... moe_destroy)."""

    def __init__(self, cfg: MoeConfig):
        self.lib = _lib.load()
        self.cfg = cfg
        h = ctypes.c_void_p()
        st = self.lib.moe_create(ctypes.byref(cfg), ctypes.byref(h))
        if st != 0:
            raise MoEError(st, self.lib.moe_last_error(None).decode())
        self.h = h

    # -- helpers
    def _check(self, st):
        if st != 0:
            raise MoEError(st, self.lib.moe_last_error(self.h).decode())

    def last_error(self) -> str:
        return self.lib.moe_last_error(self.h).decode()

    # -- ABI
    def set_router(self, layer: int, w_r: np.ndarray):
        c = self.cfg
        w = np.ascontiguousarray(w_r)
        _check_buffer("w_r", w, (4 if c.wdtype == DTYPE["fp32"] else 2) * c.n_experts * c.d, "host")
        self._check(self.lib.moe_set_router(self.h, layer, _ptr(w)))

    def register_host_experts(self, layer: int, expert: int, gate, up, down, scales=None):
        c = self.cfg
        g, u, dn = (np.ascontiguousarray(a) for a in (gate, up, down))
        for name, a in (("gate", g), ("up", u), ("down", dn)):
            _check_buffer(name, a, _weight_bytes(c.wdtype, c.d * c.d_ff), "host")
        sc = None if scales is None else np.ascontiguousarray(scales, dtype=np.uint16)
        if sc is not None:
            _check_buffer("scales", sc, 2 * (2 * c.d_ff * (c.d // 128) + c.d * (c.d_ff // 128)), "host")
        self._check(self.lib.moe_register_host_experts(self.h, layer, expert, _ptr(g), _ptr(u), _ptr(dn), _ptr(sc)))

    def _act_bytes(self, batch: int) -> int:
        c = self.cfg
        return c.n_layers * batch * c.d * (4 if c.adtype == DTYPE["fp32"] else 2)

    def decode_step(self, hidden, out, batch: int = 1, stream=None):
        """hidden, out: contiguous device tensors [n_layers x batch x d]; stream: torch.cuda.Stream or None
        (torch's current stream)."""
        import torch

        need = self._act_bytes(batch)
        _check_buffer("hidden", hidden, need, "device", self.cfg.device)
        _check_buffer("out", out, need, "device", self.cfg.device)
        if stream is None:
            stream = torch.cuda.current_stream(hidden.device)
        self._check(self.lib.moe_decode_step(self.h, _ptr(hidden), _ptr(out), batch,
                                             ctypes.c_void_p(stream.cuda_stream)))

    def decode_step_host(self, hidden, out, batch: int = 1):
        """hidden, out: host buffers (numpy arrays or CPU tensors, ideally pinned)."""
        need = self._act_bytes(batch)
        _check_buffer("hidden", hidden, need, "host")
        _check_buffer("out", out, need, "host")
        self._check(self.lib.moe_decode_step_host(self.h, _ptr(hidden), _ptr(out), batch))

    def get_residency_trace(self) -> np.ndarray:
        n_copied, n_total = ctypes.c_int64(), ctypes.c_int64()
        self.lib.moe_get_residency_trace(self.h, 0, None, 0, ctypes.byref(n_copied), ctypes.byref(n_total))
        out = np.zeros(n_total.value, dtype=TRACE_DTYPE)
        st = self.lib.moe_get_residency_trace(self.h, 0, _ptr(out), n_total.value, ctypes.byref(n_copied),
                                              ctypes.byref(n_total))
        self._check(st)
        return out[:n_copied.value]

    def get_last_routing(self):
        n = self.cfg.n_layers * self.cfg.max_batch * self.cfg.top_k
        idx = np.empty(n, dtype=np.int32)
        gate = np.empty(n, dtype=np.float32)
        self._check(self.lib.moe_get_last_routing(self.h, _ptr(idx), _ptr(gate), n))
        shape = (self.cfg.n_layers, self.cfg.max_batch, self.cfg.top_k)
        return idx.reshape(shape), gate.reshape(shape)

    def get_last_logits(self) -> np.ndarray:
        """Router logits of the last step, float32 [n_layers x max_batch x n_experts] (device schedule)."""
        c = self.cfg
        z = np.empty(c.n_layers * c.max_batch * c.n_experts, dtype=np.float32)
        self._check(self.lib.moe_get_last_logits(self.h, _ptr(z), z.size))
        return z.reshape(c.n_layers, c.max_batch, c.n_experts)

    def get_stats(self) -> dict:
        s = Stats()
        self._check(self.lib.moe_get_stats(self.h, ctypes.byref(s)))
        return {f: getattr(s, f) for f, _ in Stats._fields_}

    def reset_residency(self):
        self._check(self.lib.moe_reset_residency(self.h))

    def inject_fault(self, kind: str):
        """Test hook: arm one fault ("barrier_timeout", "copy_error" or "none") for the next step."""
        self._check(self.lib.moe_inject_fault(self.h, _lib.FAULT[kind]))

    def preload(self) -> int:
        n = ctypes.c_int64()
        self._check(self.lib.moe_preload(self.h, ctypes.byref(n)))
        return n.value

    def profile_enable(self, on: bool = True):
        self._check(self.lib.moe_profile_enable(self.h, 1 if on else 0))

    def profile_read(self) -> dict:
        arr = (KernelTime * 16)()
        n = ctypes.c_int32()
        self._check(self.lib.moe_profile_read(self.h, arr, 16, ctypes.byref(n)))
        return {arr[i].name.decode(): {"launches": arr[i].launches, "total_ms": arr[i].total_ms,
                                       "bytes": arr[i].bytes} for i in range(n.value)}

    def destroy(self):
        if getattr(self, "h", None):
            self.lib.moe_destroy(self.h)
            self.h = None

    close = destroy

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.destroy()


class Planner:
    """Residency planner (moe_planner_*): the library's host slot table driven by expert
    selections, with no GPU. step() returns the layer-step's records (TRACE_DTYPE): hits and
    misses of the used experts, then prefetch admissions (kind 2, LRU only)."""

    def __init__(self, n_layers: int, n_experts: int, cap_slots: int, policy: str = "lru"):
        self.lib = _lib.load()
        self.n_layers, self.n_experts = n_layers, n_experts
        h = ctypes.c_void_p()
        st = self.lib.moe_planner_create(n_layers, n_experts, cap_slots, _lib.POLICY[policy], ctypes.byref(h))
        if st != 0:
            raise MoEError(st, (self.lib.moe_planner_last_error(None) or b"").decode())
        self.h = h

    def _check(self, st):
        if st != 0:
            raise MoEError(st, (self.lib.moe_planner_last_error(self.h) or b"").decode())

    def preload(self) -> int:
        n = ctypes.c_int64()
        self._check(self.lib.moe_planner_preload(self.h, ctypes.byref(n)))
        return n.value

    def step(self, step: int, layer: int, experts, prefetch=(), ranks=None) -> np.ndarray:
        """ranks: the "guided" policy's [n_experts] ranks of the layer's experts in this step's
        routing (0 = highest logit; the best rank over a batch)."""
        ex = np.ascontiguousarray(np.asarray(experts, dtype=np.int32).ravel())
        pf = np.ascontiguousarray(np.asarray(prefetch, dtype=np.int32).ravel())
        rk = None
        if ranks is not None:
            rk = np.ascontiguousarray(np.asarray(ranks, dtype=np.int32).ravel())
            if rk.size != self.n_experts:
                raise ValueError(f"ranks has {rk.size} entries, expected n_experts = {self.n_experts}")
        out = np.zeros(max(1, ex.size + pf.size), dtype=TRACE_DTYPE)
        n = ctypes.c_int32()
        st = self.lib.moe_planner_step(self.h, step, layer, _ptr(ex) if ex.size else None, ex.size,
                                       _ptr(pf) if pf.size else None, pf.size, _ptr(rk), _ptr(out), out.size,
                                       ctypes.byref(n))
        recs = out[:n.value]
        if st != 0:
            err = MoEError(st, (self.lib.moe_planner_last_error(self.h) or b"").decode())
            err.records = recs
            raise err
        return recs

    def run(self, idx, ranks=None, prefetch=None, first_step: int = 0) -> dict:
        """Replay a recorded routing sequence: idx int [T x L x B x k] (or [T x L x k]) expert ids,
        as moe_get_last_routing returns them step by step; ranks [T x L x E] for the "guided"
        policy; prefetch [T x L x m] candidates (LRU only). Returns the records and per-step counts:
        {"records", "hits", "misses", "prefetches", "evictions", "hit_rate"}."""
        idx = np.asarray(idx)
        if idx.ndim == 3:
            idx = idx[:, :, None, :]
        T, L = idx.shape[0], idx.shape[1]
        if L != self.n_layers:
            raise ValueError(f"idx has {L} layers, the planner {self.n_layers}")
        recs = []
        for t in range(T):
            for l in range(L):
                recs.append(self.step(first_step + t, l, idx[t, l].ravel(),
                                      () if prefetch is None else np.asarray(prefetch[t][l]).ravel(),
                                      None if ranks is None else ranks[t][l]))
        records = np.concatenate(recs) if recs else np.zeros(0, dtype=TRACE_DTYPE)
        kind = records["kind"]
        hits, misses = int((kind == 0).sum()), int((kind == 1).sum())
        return {"records": records, "hits": hits, "misses": misses, "prefetches": int((kind == 2).sum()),
                "evictions": int((records["evicted"] >= 0).sum()), "hit_rate": hits / max(1, hits + misses)}

    def destroy(self):
        if getattr(self, "h", None):
            self.lib.moe_planner_destroy(self.h)
            self.h = None

    close = destroy

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.destroy()


def plan_caps(n_layers: int, n_experts: int, caps, idx, policy: str = "lru", ranks=None, prefetch=None,
              expert_bytes: int | None = None, preload: bool = False) -> list:
    """Capacity sweep with the residency planner: replay one recorded routing sequence (idx as for
    Planner.run) at every slot count in caps. Returns one dict per cap, in the given order: cap,
    hit_rate, misses, evictions, prefetches, misses and evictions per decode step, and, with
    expert_bytes, the host-link bytes per decode step the misses and prefetches would move."""
    T = np.asarray(idx).shape[0]
    rows = []
    for cap in caps:
        p = Planner(n_layers, n_experts, int(cap), policy)
        try:
            if preload:
                p.preload()
            r = p.run(idx, ranks=ranks, prefetch=prefetch)
        finally:
            p.destroy()
        row = {"cap": int(cap), "hit_rate": r["hit_rate"], "misses": r["misses"], "evictions": r["evictions"],
               "prefetches": r["prefetches"], "misses_per_step": r["misses"] / max(1, T),
               "evictions_per_step": r["evictions"] / max(1, T)}
        if expert_bytes is not None:
            row["link_bytes_per_step"] = (r["misses"] + r["prefetches"]) * expert_bytes / max(1, T)
        rows.append(row)
    return rows


class Decoder:
    """Chained decoder blocks around a MoE handle's layers (moe_decoder_create ... _destroy).

    The MoE handle (device schedule, max_batch 1) must outlive the decoder; decoder steps advance
    its decode steps, trace and slot group. Weights and caches use the handle's activation storage
    (float32, or bf16 bits as uint16)."""

    def __init__(self, moe: MoE, n_heads: int, n_kv_heads: int, head_dim: int, max_pos: int, eps: float = 1e-6,
                 rope_theta: float = 1e6):
        self.lib = _lib.load()
        self.moe = moe
        self.cfg = DecoderConfig(n_heads=n_heads, n_kv_heads=n_kv_heads, head_dim=head_dim, reserved=0,
                                 max_pos=max_pos, eps=eps, rope_theta=rope_theta)
        self.es = 4 if moe.cfg.adtype == DTYPE["fp32"] else 2
        h = ctypes.c_void_p()
        st = self.lib.moe_decoder_create(moe.h, ctypes.byref(self.cfg), ctypes.byref(h))
        if st != 0:
            raise MoEError(st, self.lib.moe_decoder_last_error(None).decode())
        self.h = h

    def _check(self, st):
        if st != 0:
            raise MoEError(st, self.lib.moe_decoder_last_error(self.h).decode())

    def set_layer(self, layer: int, wq, wk, wv, wo, norm_in, norm_post, norm_q, norm_k):
        """Host arrays in the activation storage: wq [n_heads*head_dim x d], wk and wv
        [n_kv_heads*head_dim x d], wo [d x n_heads*head_dim], norm_in and norm_post [d], norm_q and
        norm_k [head_dim]."""
        c, d = self.cfg, self.moe.cfg.d
        qd, kd = c.n_heads * c.head_dim, c.n_kv_heads * c.head_dim
        arrs = [np.ascontiguousarray(a) for a in (wq, wk, wv, wo, norm_in, norm_post, norm_q, norm_k)]
        sizes = (qd * d, kd * d, kd * d, d * qd, d, d, c.head_dim, c.head_dim)
        names = ("wq", "wk", "wv", "wo", "norm_in", "norm_post", "norm_q", "norm_k")
        for name, a, n in zip(names, arrs, sizes):
            _check_buffer(name, a, n * self.es, "host")
        self._check(self.lib.moe_decoder_set_layer(self.h, layer, *(_ptr(a) for a in arrs)))

    def set_cache(self, layer: int, K, V):
        """K, V: host arrays [n_kv_heads x n_pos x head_dim] in the activation storage."""
        K, V = np.ascontiguousarray(K), np.ascontiguousarray(V)
        c = self.cfg
        if K.shape != V.shape or K.ndim != 3 or K.shape[0] != c.n_kv_heads or K.shape[2] != c.head_dim:
            raise ValueError("K and V must both be [n_kv_heads x n_pos x head_dim]")
        n = K.shape[1]
        for name, a in (("K", K), ("V", V)):
            _check_buffer(name, a, c.n_kv_heads * n * c.head_dim * self.es, "host")
        self._check(self.lib.moe_decoder_set_cache(self.h, layer, _ptr(K), _ptr(V), n))

    def step(self, x_in, x_out, layer_log=None, stream=None):
        """x_in: device tensor [d] in the activation dtype; x_out: device float32 [d]; layer_log:
        None or device float32 [n_layers x 4 x d] (stream entering each layer, W_o o, MoE input,
        MoE output)."""
        import torch

        m = self.moe.cfg
        _check_buffer("x_in", x_in, m.d * self.es, "device", m.device)
        _check_buffer("x_out", x_out, m.d * 4, "device", m.device)
        if layer_log is not None:
            _check_buffer("layer_log", layer_log, m.n_layers * 4 * m.d * 4, "device", m.device)
        if stream is None:
            stream = torch.cuda.current_stream(x_in.device)
        self._check(self.lib.moe_decoder_step(self.h, _ptr(x_in), _ptr(x_out), _ptr(layer_log),
                                              ctypes.c_void_p(stream.cuda_stream)))

    @property
    def position(self) -> int:
        return int(self.lib.moe_decoder_position(self.h))

    def destroy(self):
        if getattr(self, "h", None):
            self.lib.moe_decoder_destroy(self.h)
            self.h = None

    close = destroy

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def attention_decode(q, k_cache, v_cache, n_pos: int, stream=None):
    """Grouped-query attention of one decode token (moe_attention_decode). q: device float32
    [n_heads x head_dim]; k_cache, v_cache: device bfloat16 or float32 [n_kv_heads x max_pos x
    head_dim]. Returns out, device float32 [n_heads x head_dim]."""
    import torch

    Hq, D = q.shape
    Hkv, Tmax, D2 = k_cache.shape
    if D2 != D or tuple(v_cache.shape) != tuple(k_cache.shape):
        raise ValueError("q, k_cache and v_cache shapes disagree")
    if q.dtype != torch.float32 or k_cache.dtype != v_cache.dtype or k_cache.dtype not in (torch.bfloat16,
                                                                                         torch.float32):
        raise ValueError("q must be float32, the caches both bfloat16 or both float32")
    cache_dtype = DTYPE["fp32"] if k_cache.dtype == torch.float32 else DTYPE["bf16"]
    lib = _lib.load()
    n = lib.moe_attention_scratch_floats(Hq, Hkv, D, n_pos)
    if n < 0:
        raise MoEError(-1, "moe_attention_decode does not take this shape")
    scratch = torch.empty(n, dtype=torch.float32, device=q.device)
    out = torch.empty((Hq, D), dtype=torch.float32, device=q.device)
    if stream is None:
        stream = torch.cuda.current_stream(q.device)
    st = lib.moe_attention_decode(_ptr(q), _ptr(k_cache), _ptr(v_cache), cache_dtype, Hq, Hkv, D, Tmax, n_pos,
                                  _ptr(out), _ptr(scratch), n, ctypes.c_void_p(stream.cuda_stream))
    if st != 0:
        raise MoEError(st, "moe_attention_decode rejected the arguments" if st == -1 else "launch failed")
    return out


def route_noalloc(w_r, hidden, top_k: int, renorm: bool = True, stream=None):
    """Routing without any device allocation by the library (moe_route_noalloc).

    For callers that cannot allocate device memory at routing time: the logits go to a fixed
    scratch array inside the library, and the caller passes its own outputs. w_r: contiguous
    device tensor [E x d]; hidden: contiguous device tensor [rows x d] on the same device, both
    float32 or both bfloat16. Returns (idx int32 [rows x top_k], gate float32 [rows x top_k]) as
    device tensors allocated by the caller side here (torch), never by the library. The call runs
    with hidden's device current (the library resolves its scratch array on the current device).
    """
    import torch

    if not (isinstance(w_r, torch.Tensor) and isinstance(hidden, torch.Tensor)):
        raise ValueError("w_r and hidden must be torch tensors")
    if w_r.dim() != 2 or hidden.dim() != 2:
        raise ValueError("w_r must be [E x d] and hidden [rows x d]")
    if w_r.dtype != hidden.dtype or w_r.dtype not in (torch.float32, torch.bfloat16):
        raise ValueError("w_r and hidden must both be float32 or both bfloat16")
    if not (w_r.is_cuda and hidden.is_cuda) or w_r.device != hidden.device:
        raise ValueError("w_r and hidden must be on one CUDA device")
    if not (w_r.is_contiguous() and hidden.is_contiguous()):
        raise ValueError("w_r and hidden must be contiguous")
    rows, d = hidden.shape
    E = w_r.shape[0]
    if w_r.shape[1] != d:
        raise ValueError(f"w_r has {w_r.shape[1]} columns, hidden has {d}")
    wd = DTYPE["fp32"] if w_r.dtype == torch.float32 else DTYPE["bf16"]
    with torch.cuda.device(hidden.device):
        idx = torch.empty((rows, top_k), dtype=torch.int32, device=hidden.device)
        gate = torch.empty((rows, top_k), dtype=torch.float32, device=hidden.device)
        if stream is None:
            stream = torch.cuda.current_stream(hidden.device)
        st = _lib.load().moe_route_noalloc(_ptr(w_r), _ptr(hidden), rows, E, d, top_k, 1 if renorm else 0, wd,
                                            _ptr(idx), _ptr(gate), ctypes.c_void_p(stream.cuda_stream))
    if st != 0:
        raise MoEError(st, "moe_route_noalloc rejected the arguments" if st != -3 else "moe_route_noalloc launch failed")
    return idx, gate


def build(force: bool = False) -> str:
    from .buildsys import build as _b

    return _b(force=force)


__all__ = ["MoE", "MoEError", "make_config", "expert_bytes", "pool_bytes", "TRACE_DTYPE", "build", "TraceRec",
           "route_noalloc"]
