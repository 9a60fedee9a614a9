"""fp64 CPU oracle of the capped-residency MoE decode step.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference leg may import this package. The CUDA
library never calls it and shares no code with it.

What it computes, per layer-step (paper, Section "Rotary GPU Concept", Fig. 1:
host tier, slot group, lookup table sub-module id -> slot, routing result
driving selective load and evict; the undisclosed rotary policy is replaced by
a deterministic LRU with lower-id ties):

1. routing: z = W_r h, p = softmax(z), top-k by z (ties -> lower id),
   renormalised gates g_r = p_{e_r} / sum_j p_{e_j};
2. residency: the distinct global ids needed this layer-step go through one
   LRU step (``orc_lru_step``), which yields one hit/miss record per id;
   every miss copies the expert's stored weights from the host tier into
   its slot (the oracle keeps those slot copies and computes from them);
   Policies: ``lru`` (above), ``rotary`` (``orc_rotary_step``), ``guided``
   (``orc_guided_step``: evict the resident with the worst rank in its
   layer's most recent routing, refreshed before each lookup);
2b. optional prefetch admission (``prefetch=m``, LRU only): after the step,
   the m experts each sequence's router ranks right after its top k are
   admitted into the slot group if absent (``orc_lru_admit``, records of kind
   2), evicting only experts this layer-step does not need;
3. expert FFN from the slot copy: u = silu(W_g x) * (W_u x), y_r = W_d u;
4. combine: out = sum_r g_r y_r in rank order.

All arithmetic is fp64 on exactly widened inputs (bf16/fp32 values, int4
dequantised to q * scale). ``oracle.decoder`` chains this MoE layer into a
stack of decoder blocks (attention over a KV cache, norms, residual stream). Every function here is pinned by ``tests/test_oracle_*``
against brute force, closed forms, invariants and a hand-simulated LRU trace.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "moe_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None
_lock = threading.Lock()

DTYPE_CODES = {"fp32": 0, "bf16": 1, "int4": 2}


class OrcRec(ctypes.Structure):
    _fields_ = [("step", ctypes.c_int32), ("layer", ctypes.c_int32), ("expert", ctypes.c_int32),
                ("kind", ctypes.c_int32), ("slot", ctypes.c_int32), ("evicted", ctypes.c_int32)]


REC_DTYPE = np.dtype([("step", np.int32), ("layer", np.int32), ("expert", np.int32), ("kind", np.int32),
                      ("slot", np.int32), ("evicted", np.int32)])


def compile_source(src: str, out: str) -> str:
    """Compile an oracle C source to a shared library (plain C, fp64, OpenMP over matrix rows)."""
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-fPIC", "-shared", "-o", tmp, src, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Compile liboracle.so in-tree."""
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    return compile_source(_SRC, _LIB_PATH)


def load_library(path: str):
    """Load a compiled oracle library and declare its signatures (used by lib(); tests also load
    deliberately broken builds of the same source through it)."""
    L = ctypes.CDLL(path)
    vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    L.orc_widen.argtypes = [ctypes.c_int, vp, vp, i64, i64, vp]
    L.orc_widen.restype = ctypes.c_int
    L.orc_matvec.argtypes = [vp, vp, i64, i64, vp]
    L.orc_softmax.argtypes = [vp, i64, vp]
    L.orc_topk.argtypes = [vp, i64, i32, vp, vp]
    L.orc_router.argtypes = [vp, vp, i32, i32, i32, i32, vp, vp, vp, vp, vp, vp]
    L.orc_expert_ffn.argtypes = [vp, vp, vp, vp, i32, i32, vp, vp, vp]
    L.orc_combine.argtypes = [vp, vp, i32, i32, vp]
    L.orc_lru_step.argtypes = [i64, vp, vp, vp, i64, vp, i32, i32, i32, vp]
    L.orc_lru_step.restype = i32
    L.orc_rotary_step.argtypes = [i64, vp, vp, vp, vp, vp, i32, i32, i32, vp]
    L.orc_rotary_step.restype = i32
    L.orc_lru_admit.argtypes = [i64, vp, vp, vp, i64, vp, i32, vp, i32, i32, i32, vp]
    L.orc_lru_admit.restype = i32
    L.orc_guided_step.argtypes = [i64, vp, vp, vp, vp, i64, vp, i32, i32, i32, vp]
    L.orc_guided_step.restype = i32
    f64 = ctypes.c_double
    L.orc_rmsnorm.argtypes = [vp, vp, i32, f64, vp]
    L.orc_rmsnorm.restype = None
    L.orc_rope.argtypes = [vp, i32, i64, f64, vp]
    L.orc_rope.restype = None
    L.orc_attend.argtypes = [vp, vp, vp, i32, i32, i64, i64, i32, vp, vp]
    L.orc_attend.restype = None
    return L


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = load_library(_LIB_PATH)
            _lib = L
    return _lib


def _p(a):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"], "oracle inputs must be C-contiguous"
    return ctypes.c_void_p(a.ctypes.data)


# ----------------------------------------------------------------------------------------------
# single-function entry points


def widen(dtype: str, raw: np.ndarray, rows: int, cols: int, scales: np.ndarray | None = None) -> np.ndarray:
    out = np.empty((rows, cols), dtype=np.float64)
    raw = np.ascontiguousarray(raw)
    sc = None if scales is None else np.ascontiguousarray(scales, dtype=np.uint16)
    rc = lib().orc_widen(DTYPE_CODES[dtype], _p(raw), _p(sc), rows, cols, _p(out))
    if rc != 0:
        raise ValueError("widen: bad dtype or shape")
    return out


def matvec(W: np.ndarray, x: np.ndarray) -> np.ndarray:
    W = np.ascontiguousarray(W, dtype=np.float64)
    x = np.ascontiguousarray(x, dtype=np.float64)
    y = np.empty(W.shape[0], dtype=np.float64)
    lib().orc_matvec(_p(W), _p(x), W.shape[0], W.shape[1], _p(y))
    return y


def softmax(z: np.ndarray) -> np.ndarray:
    z = np.ascontiguousarray(z, dtype=np.float64)
    p = np.empty_like(z)
    lib().orc_softmax(_p(z), z.size, _p(p))
    return p


def router(Wr: np.ndarray, h: np.ndarray, k: int, renorm: bool = True, forced_idx=None):
    """Routing of one hidden vector -> (idx int32[k], gate f64[k], z f64[E], p f64[E])."""
    Wr = np.ascontiguousarray(Wr, dtype=np.float64)
    h = np.ascontiguousarray(h, dtype=np.float64)
    E, d = Wr.shape
    idx = np.empty(k, dtype=np.int32)
    gate = np.empty(k, dtype=np.float64)
    z = np.empty(E, dtype=np.float64)
    p = np.empty(E, dtype=np.float64)
    scratch = np.empty(2 * E + (E + 7) // 8 + 1, dtype=np.float64)
    fi = None if forced_idx is None else np.ascontiguousarray(forced_idx, dtype=np.int32)
    lib().orc_router(_p(Wr), _p(h), E, d, k, 1 if renorm else 0, _p(fi), _p(idx), _p(gate), _p(z), _p(p),
                     _p(scratch))
    return idx, gate, z, p


def prefetch_candidates(z: np.ndarray, idx, m: int):
    """The m experts the router ranks highest after the selected ones: descending logit z, ties to
    the lower id, skipping the ids in idx (ranks k .. k + m - 1 when idx is the router's own top k).
    One reading of the paper's principle that residency decisions may use information produced
    during execution (Sec. 3; the routing result of Fig. 1 feeds the residency decision)."""
    sel = set(int(e) for e in idx)
    order = sorted(range(len(z)), key=lambda e: (-float(z[e]), e))
    return [e for e in order if e not in sel][:m]


def expert_ffn(Wg: np.ndarray, Wu: np.ndarray, Wd: np.ndarray, x: np.ndarray):
    """SwiGLU expert FFN in fp64 -> (y [d], u [I])."""
    Wg, Wu, Wd = (np.ascontiguousarray(a, dtype=np.float64) for a in (Wg, Wu, Wd))
    x = np.ascontiguousarray(x, dtype=np.float64)
    I, d = Wg.shape
    y = np.empty(d, dtype=np.float64)
    u = np.empty(I, dtype=np.float64)
    scratch = np.empty(3 * I, dtype=np.float64)
    lib().orc_expert_ffn(_p(Wg), _p(Wu), _p(Wd), _p(x), d, I, _p(y), _p(u), _p(scratch))
    return y, u


def combine(y: np.ndarray, gate: np.ndarray) -> np.ndarray:
    y = np.ascontiguousarray(y, dtype=np.float64)
    gate = np.ascontiguousarray(gate, dtype=np.float64)
    k, d = y.shape
    out = np.empty(d, dtype=np.float64)
    lib().orc_combine(_p(y), _p(gate), k, d, _p(out))
    return out


class LRUTable:
    """Residency state (slot group + lookup table) driven one layer-step at a time."""

    def __init__(self, n_gid: int, cap: int, n_experts: int):
        self.n_gid, self.cap, self.n_experts = n_gid, cap, n_experts
        self.slot_of = np.full(n_gid, -1, dtype=np.int32)
        self.gid_of = np.full(cap, -1, dtype=np.int32)
        self.last_use = np.full(n_gid, -1, dtype=np.int64)

    def preload(self):
        """Warm start: free slots take experts in ascending global id order until the group is full;
        they count as used before every layer-step (last use -1)."""
        free = [s for s in range(self.cap) if self.gid_of[s] < 0]
        g = 0
        for s in free:
            while g < self.n_gid and self.slot_of[g] >= 0:
                g += 1
            if g >= self.n_gid:
                break
            self.gid_of[s] = g
            self.slot_of[g] = s
            self.last_use[g] = -1
            g += 1

    def step(self, clock: int, needed, step: int) -> np.ndarray:
        needed = np.ascontiguousarray(sorted(set(int(g) for g in needed)), dtype=np.int32)
        out = np.zeros(len(needed), dtype=REC_DTYPE)
        n = lib().orc_lru_step(self.cap, _p(self.slot_of), _p(self.gid_of), _p(self.last_use), clock, _p(needed),
                               len(needed), self.n_experts, step, _p(out))
        if n < 0:
            raise RuntimeError("LRU step: capacity below the number of distinct experts in one layer-step")
        return out

    def admit(self, clock: int, pinned, admit, step: int) -> np.ndarray:
        """Prefetch admission after a layer-step (see orc_lru_admit): records of kind 2."""
        pinned = np.ascontiguousarray(sorted(set(int(g) for g in pinned)), dtype=np.int32)
        admit = np.ascontiguousarray(sorted(set(int(g) for g in admit)), dtype=np.int32)
        out = np.zeros(len(admit), dtype=REC_DTYPE)
        n = lib().orc_lru_admit(self.cap, _p(self.slot_of), _p(self.gid_of), _p(self.last_use), clock, _p(pinned),
                                len(pinned), _p(admit), len(admit), self.n_experts, step, _p(out))
        return out[:n]


class RotaryTable:
    """Residency state under the rotary slot-group policy (one reading of the paper's
    rotary residency, Fig. 1/2): a ring of slots with a hand; a miss returns to the slot it was last
    evicted from when that slot holds no expert of the step (reverse rotation), else takes the next
    such slot from the hand (forward rotation). See orc_rotary_step."""

    def __init__(self, n_gid: int, cap: int, n_experts: int):
        self.n_gid, self.cap, self.n_experts = n_gid, cap, n_experts
        self.slot_of = np.full(n_gid, -1, dtype=np.int32)
        self.gid_of = np.full(cap, -1, dtype=np.int32)
        self.prior = np.full(cap, -1, dtype=np.int32)
        self.hand = np.zeros(1, dtype=np.int64)

    def preload(self):
        """Warm start: slots 0.. take experts in ascending global id order; the hand stays at slot 0,
        so forward rotation replaces the preloaded experts first, in id order."""
        for s in range(min(self.cap, self.n_gid)):
            if self.gid_of[s] < 0:
                g = int(np.flatnonzero(self.slot_of < 0)[0])
                self.gid_of[s] = g
                self.slot_of[g] = s

    def step(self, clock: int, needed, step: int) -> np.ndarray:
        needed = np.ascontiguousarray(sorted(set(int(g) for g in needed)), dtype=np.int32)
        out = np.zeros(len(needed), dtype=REC_DTYPE)
        n = lib().orc_rotary_step(self.cap, _p(self.slot_of), _p(self.gid_of), _p(self.prior), _p(self.hand),
                                  _p(needed), len(needed), self.n_experts, step, _p(out))
        if n < 0:
            raise RuntimeError("rotary step: capacity below the number of distinct experts in one layer-step")
        return out


def route_ranks(z: np.ndarray) -> np.ndarray:
    """Rank of every expert in one routing: 0 for the highest logit, ties to the lower id."""
    order = sorted(range(len(z)), key=lambda e: (-float(z[e]), e))
    rank = np.empty(len(z), dtype=np.int32)
    rank[order] = np.arange(len(z), dtype=np.int32)
    return rank


class GuidedTable:
    """Residency state under router-guided replacement (one reading of the paper's residency
    decisions that use information produced during execution, Sec. 3): every layer keeps the rank of
    each of its experts in its most recent routing (the best rank over a batch's sequences; E before
    the layer is first routed). A miss takes the lowest free slot, else evicts the resident outside
    the layer-step's needed set with the largest rank, ties to the most recent use, then to the
    lower global id. See orc_guided_step."""

    def __init__(self, n_gid: int, cap: int, n_experts: int):
        self.n_gid, self.cap, self.n_experts = n_gid, cap, n_experts
        self.slot_of = np.full(n_gid, -1, dtype=np.int32)
        self.gid_of = np.full(cap, -1, dtype=np.int32)
        self.last_use = np.full(n_gid, -1, dtype=np.int64)
        self.rank = np.full(n_gid, n_experts, dtype=np.int32)

    preload = LRUTable.preload

    def set_layer_ranks(self, layer: int, ranks):
        E = self.n_experts
        self.rank[layer * E:(layer + 1) * E] = np.asarray(ranks, dtype=np.int32)

    def step(self, clock: int, needed, step: int) -> np.ndarray:
        needed = np.ascontiguousarray(sorted(set(int(g) for g in needed)), dtype=np.int32)
        out = np.zeros(len(needed), dtype=REC_DTYPE)
        n = lib().orc_guided_step(self.cap, _p(self.slot_of), _p(self.gid_of), _p(self.last_use), _p(self.rank),
                                  clock, _p(needed), len(needed), self.n_experts, step, _p(out))
        if n < 0:
            raise RuntimeError("guided step: capacity below the number of distinct experts in one layer-step")
        return out


TABLES = {"lru": LRUTable, "rotary": RotaryTable, "guided": GuidedTable}

# ----------------------------------------------------------------------------------------------
# the full decode step


@dataclass
class StepResult:
    out: np.ndarray | None  # f64 [L x B x d] (None when outputs were not requested)
    records: np.ndarray  # REC_DTYPE, all layer-steps of this decode step in layer order
    idx: np.ndarray  # int32 [L x B x k]
    gate: np.ndarray  # f64 [L x B x k]
    z: np.ndarray  # f64 [L x B x E] router logits


class Oracle:
    """Decode-step oracle over a stack of MoE layers with a capped slot pool.

    experts(layer, expert) -> synth.ExpertWeights (raw storage) is the host tier.
    routers[l]: raw router storage [E x d]. With keep_slot_copies the oracle copies
    an expert's stored bytes into its slot on a miss and computes from that copy.
    """

    def __init__(self, d, n_experts, top_k, d_ff, n_layers, wdtype, adtype, cap_slots, routers, experts,
                 renorm=True, keep_slot_copies=True, policy="lru", prefetch=0):
        self.d, self.E, self.k, self.I, self.L = d, n_experts, top_k, d_ff, n_layers
        self.wdtype, self.adtype, self.renorm = wdtype, adtype, renorm
        self.router_dtype = "fp32" if wdtype == "fp32" else "bf16"
        self.routers = [widen(self.router_dtype, routers[l], n_experts, d) for l in range(n_layers)]
        self.experts = experts
        self.keep = keep_slot_copies
        self.policy = policy
        if prefetch and policy != "lru":
            raise ValueError("prefetch admission is defined for the LRU policy")
        self.prefetch = prefetch  # router ranks k .. k + prefetch - 1 admitted after each layer-step
        self.table = TABLES[policy](n_layers * n_experts, cap_slots, n_experts)
        self.slots: dict[int, object] = {}
        self.token_step = 0

    @classmethod
    def for_workload(cls, wl, cap_slots=None, keep_slot_copies=True, routers=None, experts=None, renorm=True,
                     policy="lru", prefetch=0):
        import synth

        routers = routers if routers is not None else [synth.router_weights(wl, l) for l in range(wl.n_layers)]
        experts = experts if experts is not None else (lambda l, e: synth.expert_weights(wl, l, e))
        return cls(wl.d, wl.n_experts, wl.top_k, wl.d_ff, wl.n_layers, wl.wdtype, wl.adtype,
                   wl.cap_slots if cap_slots is None else cap_slots, routers, experts, renorm=renorm,
                   keep_slot_copies=keep_slot_copies, policy=policy, prefetch=prefetch)

    def reset(self):
        self.table = TABLES[self.policy](self.table.n_gid, self.table.cap, self.E)
        self.slots = {}
        self.token_step = 0

    def preload(self):
        """Warm start (see LRUTable.preload), copying each preloaded expert into its slot."""
        self.table.preload()
        if self.keep:
            for s, g in enumerate(self.table.gid_of):
                if g >= 0 and s not in self.slots:
                    l, e = divmod(int(g), self.E)
                    self.slots[s] = (int(g), _copy_expert(self.experts(l, e)))

    def _widen_expert(self, w):
        d, I, dt = self.d, self.I, self.wdtype
        Wg = widen(dt, w.gate, I, d, w.s_gate)
        Wu = widen(dt, w.up, I, d, w.s_up)
        Wd = widen(dt, w.down, d, I, w.s_down)
        return Wg, Wu, Wd

    def moe_layer(self, layer: int, h_raw: np.ndarray, forced_idx=None):
        """One layer's output for one hidden vector, reading the host tier directly.

        Same definition as decode_step without the slot group; the cap invariant (outputs do
        not depend on residency) is what lets sampled outputs of large runs be checked this way.
        Returns (out f64 [d], idx, gate).
        """
        import synth

        h = synth.act_to_f64(np.asarray(h_raw), self.adtype)
        idx, gate, _, _ = router(self.routers[layer], h, self.k, self.renorm, forced_idx)
        ys = np.empty((self.k, self.d), dtype=np.float64)
        for rk in range(self.k):
            Wg, Wu, Wd = self._widen_expert(self.experts(layer, int(idx[rk])))
            ys[rk], _ = expert_ffn(Wg, Wu, Wd, h)
        return combine(ys, gate), idx, gate

    def decode_step(self, hidden_raw: np.ndarray, compute_out: bool = True, forced_idx=None,
                    forced_ranks=None) -> StepResult:
        """One decode step over all layers. hidden_raw: raw activation storage [L x B x d].
        forced_idx [L x B x k] / forced_ranks [L x E] replace the routing's choices and the guided
        policy's ranks (to replay a run whose fp32 logits swapped near-equal experts)."""
        import synth

        L, B = hidden_raw.shape[0], hidden_raw.shape[1]
        assert L == self.L and hidden_raw.shape[2] == self.d
        h = synth.act_to_f64(hidden_raw, self.adtype)
        idx = np.empty((L, B, self.k), dtype=np.int32)
        gate = np.empty((L, B, self.k), dtype=np.float64)
        z = np.empty((L, B, self.E), dtype=np.float64)
        out = np.zeros((L, B, self.d), dtype=np.float64) if compute_out else None
        recs = []
        for l in range(L):
            o, idx[l], gate[l], z[l], r = self.layer_step(l, h[l], compute_out,
                                                          None if forced_idx is None else forced_idx[l],
                                                          None if forced_ranks is None else forced_ranks[l])
            if compute_out:
                out[l] = o
            recs.append(r)
        self.token_step += 1
        return StepResult(out, np.concatenate(recs), idx, gate, z)

    def layer_step(self, l: int, h: np.ndarray, compute_out: bool = True, forced_idx=None, forced_ranks=None):
        """Layer l of the current decode step on fp64 inputs h [B x d]: routing, one residency step,
        expert FFNs from the slot copies and the combine. The clock is token_step * L + l; the
        caller advances token_step once per decode step (decode_step does).
        Returns (out [B x d] or None, idx [B x k], gate [B x k], z [B x E], records)."""
        B = h.shape[0]
        idx = np.empty((B, self.k), dtype=np.int32)
        gate = np.empty((B, self.k), dtype=np.float64)
        z = np.empty((B, self.E), dtype=np.float64)
        clock = self.token_step * self.L + l
        for b in range(B):
            fi = None if forced_idx is None else forced_idx[b]
            idx[b], gate[b], z[b], _ = router(self.routers[l], h[b], self.k, self.renorm, fi)
        needed = sorted(set(int(l * self.E + e) for e in idx.ravel()))
        if self.policy == "guided":
            ranks = np.min([route_ranks(z[b]) for b in range(B)], axis=0) if forced_ranks is None else forced_ranks
            self.table.set_layer_ranks(l, ranks)
        r = self.table.step(clock, needed, self.token_step)
        if self.prefetch:
            admit = set()
            for b in range(B):
                admit.update(l * self.E + e for e in prefetch_candidates(z[b], idx[b], self.prefetch))
            r = np.concatenate([r, self.table.admit(clock, needed, sorted(admit - set(needed)), self.token_step)])
        for rec in r:
            if rec["kind"] in (1, 2):
                gid = int(l * self.E + rec["expert"])
                if self.keep:
                    w = self.experts(l, int(rec["expert"]))
                    self.slots[int(rec["slot"])] = (gid, _copy_expert(w))
        out = None
        if compute_out:
            out = np.zeros((B, self.d), dtype=np.float64)
            cache = {}
            for b in range(B):
                ys = np.empty((self.k, self.d), dtype=np.float64)
                for rk in range(self.k):
                    e = int(idx[b, rk])
                    gid = l * self.E + e
                    if gid not in cache:
                        if self.keep:
                            slot = int(self.table.slot_of[gid])
                            held_gid, w = self.slots[slot]
                            assert held_gid == gid, "slot holds another expert"
                        else:
                            w = self.experts(l, e)
                        cache[gid] = self._widen_expert(w)
                    Wg, Wu, Wd = cache[gid]
                    ys[rk], _ = expert_ffn(Wg, Wu, Wd, h[b])
                out[b] = combine(ys, gate[b])
        return out, idx, gate, z, r


def _copy_expert(w):
    import copy

    c = copy.copy(w)
    for f in ("gate", "up", "down", "s_gate", "s_up", "s_down"):
        v = getattr(w, f)
        setattr(c, f, None if v is None else v.copy())
    return c
