"""The Python binding refuses, before calling the library, buffers the library would read or write
past their end or on the wrong side of the host/device boundary (the C calls copy fixed sizes
from the pointers they are given)."""
import numpy as np
import pytest
import torch

import paper_2605_29135_gb300 as P


def _handleless(wdtype="bf16", adtype="bf16", d=256, E=8, k=2, I=128, L=2, max_batch=4):
    m = P.MoE.__new__(P.MoE)
    m.cfg = P.make_config(d, E, k, I, L, wdtype, adtype, cap_slots=4, max_batch=max_batch)
    m.lib = None  # any call that reached the library would fail loudly
    m.h = None
    return m


def test_decode_step_needs_device_buffers_of_the_full_size():
    m = _handleless()
    cpu = torch.zeros((2, 4, 256), dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="cuda:0"):
        m.decode_step(cpu, cpu, batch=4)


def test_decode_step_host_checks_sizes_and_side():
    m = _handleless()
    ok = np.zeros((2, 4, 256), dtype=np.uint16)
    small = np.zeros((2, 3, 256), dtype=np.uint16)
    with pytest.raises(ValueError, match="bytes"):
        m.decode_step_host(small, ok, batch=4)
    with pytest.raises(ValueError, match="bytes"):
        m.decode_step_host(ok, small, batch=4)
    with pytest.raises(ValueError, match="contiguous"):
        m.decode_step_host(np.zeros((2, 4, 512), dtype=np.uint16)[:, :, ::2], ok, batch=4)


def test_router_and_expert_registration_check_sizes():
    m = _handleless()
    with pytest.raises(ValueError, match="w_r"):
        m.set_router(0, np.zeros((8, 255), dtype=np.uint16))
    full = np.zeros((128, 256), dtype=np.uint16)
    with pytest.raises(ValueError, match="down"):
        m.register_host_experts(0, 0, full, full, np.zeros((256, 127), dtype=np.uint16))
    m4 = _handleless(wdtype="int4")
    q = np.zeros((128, 128), dtype=np.uint8)  # int4: two elements per byte
    qd = np.zeros((256, 64), dtype=np.uint8)
    with pytest.raises(ValueError, match="scales"):
        m4.register_host_experts(0, 0, q, q, qd, np.zeros(10, dtype=np.uint16))


def test_none_buffers_are_refused():
    m = _handleless()
    with pytest.raises(ValueError, match="None"):
        m.decode_step_host(None, np.zeros(4096, dtype=np.uint16), batch=1)


def test_route_noalloc_refuses_mismatched_or_host_tensors_before_calling_the_library():
    w = torch.zeros((8, 256), dtype=torch.bfloat16)
    h = torch.zeros((2, 256), dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="CUDA device"):
        P.route_noalloc(w, h, 2)
    with pytest.raises(ValueError, match="float32 or both bfloat16"):
        P.route_noalloc(w, h.float(), 2)
    with pytest.raises(ValueError, match="float32 or both bfloat16"):
        P.route_noalloc(w.half(), h.half(), 2)
    with pytest.raises(ValueError, match=r"\[E x d\]"):
        P.route_noalloc(w, h[0], 2)
    with pytest.raises(ValueError, match="torch tensors"):
        P.route_noalloc(np.zeros((8, 256), np.float32), h, 2)
