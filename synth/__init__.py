"""Seeded synthetic inputs for the capped-residency MoE decode step.

Shared by the fp64 oracle (``oracle/``) and the CUDA path: this module is the
single source of input values and holds none of the decode step's arithmetic.
Weights are N(0, std = 1/sqrt(fan_in)) in fp32 from a counter-based generator
(SplitMix64 hash + Box-Muller), then stored as fp32, bf16 (round to nearest
even) or symmetric int4 with group size 128 along the input dimension and bf16
scales. Hidden states are AR(1) streams h_t = rho h_{t-1} + sqrt(1-rho^2) eps_t
computed in fp64 and rounded to the activation dtype (fp64 -> fp32 -> bf16).

The MoE setting these inputs stand in for is the paper's Section "Rotary GPU
Concept" (sub-modules = experts held in a host tier, a routing result driving
residency); the synthetic shapes follow a Qwen3-30B-A3B-class MoE layer.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_LIB_PATH = os.path.join(_HERE, "libsynth.so")
_lib = None
_lock = threading.Lock()

WDTYPES = {"fp32": 0, "bf16": 1, "int4": 2}
HIDDEN_STREAM_TAG = 1 << 60


def build(force: bool = False) -> str:
    """Compile libsynth.so in-tree with the host C compiler."""
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-ffp-contract=off", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB_PATH)
            u64, i64, vp = ctypes.c_uint64, ctypes.c_int64, ctypes.c_void_p
            L.synth_key.argtypes = [u64, u64]
            L.synth_key.restype = u64
            L.synth_hash.argtypes = [u64, u64]
            L.synth_hash.restype = u64
            L.synth_normal.argtypes = [u64, u64, u64, i64, ctypes.c_float, vp]
            L.synth_normal.restype = None
            L.synth_f32_to_bf16.argtypes = [vp, vp, i64]
            L.synth_f64_to_f32.argtypes = [vp, vp, i64]
            L.synth_f64_to_bf16.argtypes = [vp, vp, i64]
            L.synth_ar1.argtypes = [u64, u64, i64, i64, ctypes.c_double, vp, vp]
            L.synth_quant_int4_g128.argtypes = [vp, i64, i64, vp, vp]
            L.synth_quant_int4_g128.restype = ctypes.c_int
            L.synth_weight_stream.argtypes = [i64, i64, i64]
            L.synth_weight_stream.restype = u64
            L.synth_weight.argtypes = [u64, i64, i64, i64, i64, i64, ctypes.c_int, vp, vp, vp]
            L.synth_weight.restype = ctypes.c_int
            _lib = L
    return _lib


def _p(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return ctypes.c_void_p(a.ctypes.data)


# ----------------------------------------------------------------------------------------------
# primitive generators


def normal(seed: int, stream: int, start: int, n: int, std: float = 1.0) -> np.ndarray:
    out = np.empty(n, dtype=np.float32)
    lib().synth_normal(seed, stream, start, n, std, _p(out))
    return out


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    lib().synth_f32_to_bf16(_p(x), _p(out), x.size)
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Decode bf16 bit patterns to float32 (exact)."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def quant_int4_g128(w: np.ndarray):
    """Symmetric int4 g128 quantisation of a fp32 [rows x cols] matrix -> (packed uint8, bf16 scale bits)."""
    w = np.ascontiguousarray(w, dtype=np.float32)
    rows, cols = w.shape
    q = np.empty((rows, cols // 2), dtype=np.uint8)
    s = np.empty((rows, cols // 128), dtype=np.uint16)
    rc = lib().synth_quant_int4_g128(_p(w), rows, cols, _p(q), _p(s))
    if rc != 0:
        raise ValueError("cols must be a multiple of 128")
    return q, s


def ar1(seed: int, stream: int, T: int, d: int, rho: float) -> np.ndarray:
    """fp64 AR(1) stream [T x d] with unit stationary variance."""
    out = np.empty((T, d), dtype=np.float64)
    scratch = np.empty(d, dtype=np.float32)
    lib().synth_ar1(seed, stream, T, d, rho, _p(out), _p(scratch))
    return out


# ----------------------------------------------------------------------------------------------
# workloads


@dataclass(frozen=True)
class Workload:
    """One synthetic MoE decode workload (all values seeded)."""

    name: str
    d: int  # hidden size
    n_experts: int  # E per layer
    top_k: int
    d_ff: int  # SwiGLU intermediate size I
    n_layers: int
    wdtype: str  # expert weight storage: fp32 | bf16 | int4
    adtype: str  # activation dtype: fp32 | bf16
    tokens: int  # decode steps in the full run
    batch: int
    rho: float
    cap_slots: int
    weight_seed: int = 0
    description: str = field(default="", compare=False)

    @property
    def router_dtype(self) -> str:
        return "fp32" if self.wdtype == "fp32" else "bf16"

    @property
    def n_gid(self) -> int:
        return self.n_layers * self.n_experts

    def expert_bytes(self) -> int:
        return expert_bytes(self.d, self.d_ff, self.wdtype)

    def router_bytes(self) -> int:
        return self.n_experts * self.d * (4 if self.router_dtype == "fp32" else 2)

    def replace(self, **kw) -> "Workload":
        from dataclasses import replace

        return replace(self, **kw)


def expert_bytes(d: int, I: int, wdtype: str) -> int:
    n = 3 * d * I
    if wdtype == "fp32":
        return 4 * n
    if wdtype == "bf16":
        return 2 * n
    if wdtype == "int4":
        return n // 2 + 2 * (n // 128)
    raise ValueError(wdtype)


_CAP_BYTES = 6_000_000_000  # the 6 GB expert pool of the capped stack workloads

WORKLOADS = {
    "tiny_fp32": Workload("tiny_fp32", d=256, n_experts=8, top_k=2, d_ff=128, n_layers=1, wdtype="fp32",
                          adtype="fp32", tokens=64, batch=1, rho=0.9, cap_slots=4,
                          description="tiny single MoE layer, fp32, 64 tokens AR(1) rho=0.9, 4 slots"),
    "layer_bf16": Workload("layer_bf16", d=2048, n_experts=128, top_k=8, d_ff=768, n_layers=1, wdtype="bf16",
                           adtype="bf16", tokens=2048, batch=1, rho=0.8, cap_slots=32,
                           description="one Qwen3-30B-A3B-shaped MoE layer, bf16, 2048 tokens, 32 of 128 slots"),
    "stack48_bf16": Workload("stack48_bf16", d=2048, n_experts=128, top_k=8, d_ff=768, n_layers=48, wdtype="bf16",
                             adtype="bf16", tokens=2048, batch=1, rho=0.8,
                             cap_slots=_CAP_BYTES // expert_bytes(2048, 768, "bf16"),
                             description="48-layer bf16 stack, 6144 experts pinned on host, 6 GB pool (635 slots)"),
    "stack48_int4": Workload("stack48_int4", d=2048, n_experts=128, top_k=8, d_ff=768, n_layers=48, wdtype="int4",
                             adtype="bf16", tokens=2048, batch=1, rho=0.8,
                             cap_slots=_CAP_BYTES // expert_bytes(2048, 768, "int4"),
                             description="48-layer int4 g128 stack, 6 GB pool (2466 slots)"),
    "stack48_batch64": Workload("stack48_batch64", d=2048, n_experts=128, top_k=8, d_ff=768, n_layers=48,
                                wdtype="bf16", adtype="bf16", tokens=512, batch=64, rho=0.8,
                                cap_slots=_CAP_BYTES // expert_bytes(2048, 768, "bf16"),
                                description="48-layer bf16 stack, 64 sequences, 512 steps, 6 GB pool"),
}


def router_weights(wl: Workload, layer: int) -> np.ndarray:
    """Router matrix W_r [E x d], raw storage: float32, or bf16 bits as uint16."""
    E, d = wl.n_experts, wl.d
    code = WDTYPES[wl.router_dtype]
    out = np.empty((E, d), dtype=np.float32 if code == 0 else np.uint16)
    tmp = np.empty(E * d, dtype=np.float32)
    rc = lib().synth_weight(wl.weight_seed, layer, 0, 3, E, d, code, _p(out), None, _p(tmp))
    assert rc == 0
    return out


@dataclass
class ExpertWeights:
    """Raw storage of one expert: gate/up [I x d], down [d x I] (out x in, row-major).

    fp32: float32 arrays; bf16: uint16 bit arrays; int4: packed uint8 [rows x in/2] plus
    bf16 scale bits [rows x in/128] per matrix (scales = concat(gate, up, down) when flat).
    """

    gate: np.ndarray
    up: np.ndarray
    down: np.ndarray
    s_gate: np.ndarray | None = None
    s_up: np.ndarray | None = None
    s_down: np.ndarray | None = None

    def scales_flat(self) -> np.ndarray | None:
        if self.s_gate is None:
            return None
        return np.concatenate([self.s_gate.ravel(), self.s_up.ravel(), self.s_down.ravel()])


def expert_weights(wl: Workload, layer: int, expert: int, tmp: np.ndarray | None = None) -> ExpertWeights:
    d, I = wl.d, wl.d_ff
    code = WDTYPES[wl.wdtype]
    if tmp is None:
        tmp = np.empty(d * I, dtype=np.float32)
    mats = []
    for m, (rows, cols) in enumerate(((I, d), (I, d), (d, I))):
        if code == 0:
            out = np.empty((rows, cols), dtype=np.float32)
        elif code == 1:
            out = np.empty((rows, cols), dtype=np.uint16)
        else:
            out = np.empty((rows, cols // 2), dtype=np.uint8)
        sc = np.empty((rows, cols // 128), dtype=np.uint16) if code == 2 else None
        rc = lib().synth_weight(wl.weight_seed, layer, expert, m, rows, cols, code, _p(out),
                                None if sc is None else _p(sc), _p(tmp))
        assert rc == 0
        mats.append((out, sc))
    return ExpertWeights(mats[0][0], mats[1][0], mats[2][0], mats[0][1], mats[1][1], mats[2][1])


def hidden_stream(wl: Workload, layer: int, seq: int = 0, tokens: int | None = None) -> np.ndarray:
    """Hidden inputs of one layer (and sequence) for all decode steps, raw activation storage.

    AR(1) with the workload's rho, random stream keyed by seed = layer and the sequence index.
    fp32 workloads: float32 [T x d]; bf16 workloads: bf16 bits uint16 [T x d].
    """
    T = wl.tokens if tokens is None else tokens
    h = ar1(layer, HIDDEN_STREAM_TAG | seq, T, wl.d, wl.rho)
    if wl.adtype == "fp32":
        out = np.empty(h.shape, dtype=np.float32)
        lib().synth_f64_to_f32(_p(h), _p(out), h.size)
    else:
        out = np.empty(h.shape, dtype=np.uint16)
        lib().synth_f64_to_bf16(_p(h), _p(out), h.size)
    return out


def hidden_all(wl: Workload, tokens: int | None = None, threads: int | None = None) -> np.ndarray:
    """Hidden inputs for every decode step: raw [T x L x B x d] in the layout a decode step takes."""
    T = wl.tokens if tokens is None else tokens
    dt = np.float32 if wl.adtype == "fp32" else np.uint16
    out = np.empty((T, wl.n_layers, wl.batch, wl.d), dtype=dt)

    def one(ls):
        l, s = ls
        out[:, l, s, :] = hidden_stream(wl, l, s, T)

    jobs = [(l, s) for l in range(wl.n_layers) for s in range(wl.batch)]
    with ThreadPoolExecutor(max_workers=threads or os.cpu_count()) as ex:
        list(ex.map(one, jobs))
    return out


def act_to_f64(raw: np.ndarray, adtype: str) -> np.ndarray:
    """Decode raw activation storage to float64 (exact widening)."""
    if adtype == "fp32":
        return raw.astype(np.float64)
    return bf16_bits_to_f32(raw).astype(np.float64)


# ----------------------------------------------------------------------------------------------
# decoder blocks around the MoE layer (attention with a KV cache, norms, a residual stream)

# matrix ids of a layer's attention weights in the weight streams (experts use 0-2, the router 3)
_ATTN_MATRIX = {"wq": 4, "wk": 5, "wv": 6, "wo": 7}
_NORM_MATRIX = {"in": 8, "post": 9, "q": 10, "k": 11}
_KV_MATRIX = {"k": 12, "v": 13}
TOKEN_INPUT_SEED = 1 << 20  # seed of the token-input streams (layers use seeds 0..L-1)


@dataclass(frozen=True)
class DecoderWorkload:
    """A chained stack of decoder blocks: per layer, x += W_o attn(...) then x += MoE(...).

    moe: the MoE layer's workload (its n_layers is the stack depth, its wdtype/adtype the storage
    of every weight and of the KV cache). ctx: positions already in the KV cache when the first
    decode token arrives (a seeded N(0, 1) prefix). The attention follows a Qwen3-MoE-class block:
    grouped-query heads with per-head RMSNorm on q and k and rotary positions.
    """

    name: str
    moe: Workload
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ctx: int
    eps: float = 1e-6
    rope_theta: float = 1e6
    norm_std: float = 0.1  # RMSNorm weights are 1 + N(0, norm_std^2)
    description: str = field(default="", compare=False)

    def replace(self, **kw) -> "DecoderWorkload":
        from dataclasses import replace

        return replace(self, **kw)


DECODERS = {
    "tiny_block_fp32": DecoderWorkload(
        "tiny_block_fp32", WORKLOADS["tiny_fp32"].replace(n_layers=2, tokens=8, cap_slots=6),
        n_heads=4, n_kv_heads=2, head_dim=64, ctx=24,
        description="2 tiny fp32 decoder blocks (d=256, 4 query / 2 kv heads of 64, E=8, top-2), 24 cached positions"),
    "block48_bf16": DecoderWorkload(
        "block48_bf16", WORKLOADS["stack48_bf16"], n_heads=32, n_kv_heads=4, head_dim=128, ctx=4095,
        description="48 Qwen3-30B-A3B-class decoder blocks, bf16, 4095 cached positions (context 4096), 6 GB pool"),
}


def _store(x: np.ndarray, dtype: str) -> np.ndarray:
    """fp32 values -> raw storage of dtype (float32, or bf16 bits)."""
    if dtype == "fp32":
        return np.ascontiguousarray(x, dtype=np.float32)
    return f32_to_bf16_bits(x)


def attention_weights(dw: DecoderWorkload, layer: int) -> dict:
    """Raw storage of one layer's attention and norm weights: wq [Hq*Dh x d], wk and wv
    [Hkv*Dh x d], wo [d x Hq*Dh] (out x in, N(0, 1/fan_in)); norm_in and norm_post [d], norm_q and
    norm_k [Dh] (1 + N(0, norm_std^2)). fp32 workloads: float32; otherwise bf16 bits."""
    wl = dw.moe
    dt = "fp32" if wl.wdtype == "fp32" else "bf16"
    code = WDTYPES[dt]
    d, qd, kd = wl.d, dw.n_heads * dw.head_dim, dw.n_kv_heads * dw.head_dim
    out = {}
    for name, (rows, cols) in (("wq", (qd, d)), ("wk", (kd, d)), ("wv", (kd, d)), ("wo", (d, qd))):
        w = np.empty((rows, cols), dtype=np.float32 if code == 0 else np.uint16)
        tmp = np.empty(rows * cols, dtype=np.float32)
        rc = lib().synth_weight(wl.weight_seed, layer, 0, _ATTN_MATRIX[name], rows, cols, code, _p(w), None, _p(tmp))
        assert rc == 0
        out[name] = w
    for name, n in (("in", d), ("post", d), ("q", dw.head_dim), ("k", dw.head_dim)):
        stream = lib().synth_weight_stream(layer, 0, _NORM_MATRIX[name])
        out["norm_" + name] = _store(1.0 + normal(wl.weight_seed, stream, 0, n, dw.norm_std), dt)
    return out


def kv_prefix(dw: DecoderWorkload, layer: int) -> tuple[np.ndarray, np.ndarray]:
    """The KV cache contents of one layer before the first decode token: K and V [Hkv x ctx x Dh],
    N(0, 1), in the activation storage (float32, or bf16 bits)."""
    wl = dw.moe
    n = dw.n_kv_heads * dw.ctx * dw.head_dim
    kv = []
    for name in ("k", "v"):
        stream = lib().synth_weight_stream(layer, 0, _KV_MATRIX[name])
        kv.append(_store(normal(wl.weight_seed, stream, 0, n, 1.0), wl.adtype).reshape(
            dw.n_kv_heads, dw.ctx, dw.head_dim))
    return kv[0], kv[1]


def token_inputs(dw: DecoderWorkload, tokens: int | None = None, seq: int = 0) -> np.ndarray:
    """The residual stream entering layer 0 at each decode token: an AR(1) stream (the MoE
    workload's rho) [T x d] in the activation storage."""
    wl = dw.moe
    T = wl.tokens if tokens is None else tokens
    h = ar1(TOKEN_INPUT_SEED, HIDDEN_STREAM_TAG | seq, T, wl.d, wl.rho)
    if wl.adtype == "fp32":
        out = np.empty(h.shape, dtype=np.float32)
        lib().synth_f64_to_f32(_p(h), _p(out), h.size)
    else:
        out = np.empty(h.shape, dtype=np.uint16)
        lib().synth_f64_to_bf16(_p(h), _p(out), h.size)
    return out
