"""ctypes declarations of libmoe.so (the C ABI declared in include/moe.h).

Argument marshalling only: every step of the decode path runs inside the library. Loading
fails loudly if the library has not been built; there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
import threading

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libmoe.so")

MOE_OK = 0
STATUS = {0: "MOE_OK", -1: "MOE_ERR_INVALID", -2: "MOE_ERR_OOM", -3: "MOE_ERR_CUDA", -4: "MOE_ERR_CAPACITY",
          -5: "MOE_ERR_NOT_REGISTERED", -6: "MOE_ERR_TIMEOUT", -7: "MOE_ERR_TRACE_OVERFLOW"}
DTYPE = {"fp32": 0, "bf16": 1, "int4": 2}
SCHEDULE = {"device": 0, "host_copy_engine": 1}
BATCHED_PATH = {"auto": 0, "cuda_cores": 1}
POLICY = {"lru": 0, "rotary": 1, "guided": 2}
FAULT = {"none": 0, "barrier_timeout": 1, "copy_error": 2}

# Every function the header declares (checked by the CPU test suite).
EXPORTS = ["moe_expert_bytes", "moe_pool_bytes", "moe_create", "moe_set_router", "moe_register_host_experts",
           "moe_decode_step", "moe_decode_step_host", "moe_get_residency_trace", "moe_get_last_routing",
           "moe_get_stats", "moe_reset_residency", "moe_profile_enable", "moe_profile_read", "moe_last_error",
           "moe_destroy", "moe_route_noalloc", "moe_preload", "moe_inject_fault", "moe_planner_create",
           "moe_planner_preload", "moe_planner_step", "moe_planner_last_error", "moe_planner_destroy",
           "moe_get_last_logits", "moe_attention_scratch_floats", "moe_attention_decode", "moe_decoder_create",
           "moe_decoder_set_layer", "moe_decoder_set_cache", "moe_decoder_step", "moe_decoder_position",
           "moe_decoder_last_error", "moe_decoder_destroy"]


class MoeConfig(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int32), ("n_experts", ctypes.c_int32), ("top_k", ctypes.c_int32),
                ("d_ff", ctypes.c_int32), ("n_layers", ctypes.c_int32), ("max_batch", ctypes.c_int32),
                ("wdtype", ctypes.c_int32), ("adtype", ctypes.c_int32), ("cap_slots", ctypes.c_int64),
                ("cap_bytes", ctypes.c_int64), ("renorm", ctypes.c_int32), ("device", ctypes.c_int32),
                ("device_pool", ctypes.c_void_p), ("trace_capacity", ctypes.c_int64), ("schedule", ctypes.c_int32),
                ("miss_ctas", ctypes.c_int32), ("batched_path", ctypes.c_int32), ("policy", ctypes.c_int32),
                ("lookahead", ctypes.c_int32)]


class DecoderConfig(ctypes.Structure):
    _fields_ = [("n_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("reserved", ctypes.c_int32), ("max_pos", ctypes.c_int64), ("eps", ctypes.c_double),
                ("rope_theta", ctypes.c_double)]


class TraceRec(ctypes.Structure):
    _fields_ = [("step", ctypes.c_int32), ("layer", ctypes.c_int32), ("expert", ctypes.c_int32),
                ("kind", ctypes.c_int32), ("slot", ctypes.c_int32), ("evicted", ctypes.c_int32)]


class Stats(ctypes.Structure):
    _fields_ = [("steps", ctypes.c_int64), ("layer_steps", ctypes.c_int64), ("hits", ctypes.c_int64),
                ("misses", ctypes.c_int64), ("evictions", ctypes.c_int64), ("miss_bytes", ctypes.c_int64)]


class KernelTime(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 32), ("launches", ctypes.c_int64), ("total_ms", ctypes.c_double),
                ("bytes", ctypes.c_int64)]


_lib = None
_lock = threading.Lock()


def load(path: str | None = None):
    """Load libmoe.so and declare its signatures. Raises if the library is missing."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"libmoe.so is not built ({p}); run `python -m paper_2605_29135_gb300.buildsys` "
                               "or __graft_entry__.build()")
        L = ctypes.CDLL(p)
        vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        cfgp = ctypes.POINTER(MoeConfig)
        L.moe_expert_bytes.argtypes = [cfgp]
        L.moe_expert_bytes.restype = i64
        L.moe_pool_bytes.argtypes = [cfgp]
        L.moe_pool_bytes.restype = i64
        L.moe_create.argtypes = [cfgp, ctypes.POINTER(vp)]
        L.moe_create.restype = ctypes.c_int
        L.moe_set_router.argtypes = [vp, i32, vp]
        L.moe_set_router.restype = ctypes.c_int
        L.moe_register_host_experts.argtypes = [vp, i32, i32, vp, vp, vp, vp]
        L.moe_register_host_experts.restype = ctypes.c_int
        L.moe_decode_step.argtypes = [vp, vp, vp, i32, vp]
        L.moe_decode_step.restype = ctypes.c_int
        L.moe_decode_step_host.argtypes = [vp, vp, vp, i32]
        L.moe_decode_step_host.restype = ctypes.c_int
        L.moe_get_residency_trace.argtypes = [vp, i64, vp, i64, ctypes.POINTER(i64), ctypes.POINTER(i64)]
        L.moe_get_residency_trace.restype = ctypes.c_int
        L.moe_get_last_routing.argtypes = [vp, vp, vp, i64]
        L.moe_get_last_routing.restype = ctypes.c_int
        L.moe_get_stats.argtypes = [vp, ctypes.POINTER(Stats)]
        L.moe_get_stats.restype = ctypes.c_int
        L.moe_reset_residency.argtypes = [vp]
        L.moe_reset_residency.restype = ctypes.c_int
        L.moe_profile_enable.argtypes = [vp, i32]
        L.moe_profile_enable.restype = ctypes.c_int
        L.moe_profile_read.argtypes = [vp, ctypes.POINTER(KernelTime), i32, ctypes.POINTER(i32)]
        L.moe_profile_read.restype = ctypes.c_int
        L.moe_last_error.argtypes = [vp]
        L.moe_last_error.restype = ctypes.c_char_p
        L.moe_destroy.argtypes = [vp]
        L.moe_destroy.restype = None
        L.moe_route_noalloc.argtypes = [vp, vp, i32, i32, i32, i32, i32, i32, vp, vp, vp]
        L.moe_route_noalloc.restype = ctypes.c_int
        L.moe_preload.argtypes = [vp, ctypes.POINTER(i64)]
        L.moe_preload.restype = ctypes.c_int
        L.moe_inject_fault.argtypes = [vp, i32]
        L.moe_inject_fault.restype = ctypes.c_int
        L.moe_planner_create.argtypes = [i32, i32, i64, i32, ctypes.POINTER(vp)]
        L.moe_planner_create.restype = ctypes.c_int
        L.moe_planner_preload.argtypes = [vp, ctypes.POINTER(i64)]
        L.moe_planner_preload.restype = ctypes.c_int
        L.moe_planner_step.argtypes = [vp, i64, i32, vp, i32, vp, i32, vp, vp, i32, ctypes.POINTER(i32)]
        L.moe_planner_step.restype = ctypes.c_int
        L.moe_planner_last_error.argtypes = [vp]
        L.moe_planner_last_error.restype = ctypes.c_char_p
        L.moe_get_last_logits.argtypes = [vp, vp, i64]
        L.moe_get_last_logits.restype = ctypes.c_int
        L.moe_attention_scratch_floats.argtypes = [i32, i32, i32, i64]
        L.moe_attention_scratch_floats.restype = i64
        L.moe_attention_decode.argtypes = [vp, vp, vp, i32, i32, i32, i32, i64, i64, vp, vp, i64, vp]
        L.moe_attention_decode.restype = ctypes.c_int
        L.moe_decoder_create.argtypes = [vp, ctypes.POINTER(DecoderConfig), ctypes.POINTER(vp)]
        L.moe_decoder_create.restype = ctypes.c_int
        L.moe_decoder_set_layer.argtypes = [vp, i32, vp, vp, vp, vp, vp, vp, vp, vp]
        L.moe_decoder_set_layer.restype = ctypes.c_int
        L.moe_decoder_set_cache.argtypes = [vp, i32, vp, vp, i64]
        L.moe_decoder_set_cache.restype = ctypes.c_int
        L.moe_decoder_step.argtypes = [vp, vp, vp, vp, vp]
        L.moe_decoder_step.restype = ctypes.c_int
        L.moe_decoder_position.argtypes = [vp]
        L.moe_decoder_position.restype = i64
        L.moe_decoder_last_error.argtypes = [vp]
        L.moe_decoder_last_error.restype = ctypes.c_char_p
        L.moe_decoder_destroy.argtypes = [vp]
        L.moe_decoder_destroy.restype = None
        L.moe_planner_destroy.argtypes = [vp]
        L.moe_planner_destroy.restype = None
        _lib = L
        return L
