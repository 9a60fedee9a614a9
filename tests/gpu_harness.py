"""Helpers shared by the GPU parity tests: run the CUDA path through the C ABI, run the oracle
on the same seeded inputs, and compare them under the stated tolerances."""
from __future__ import annotations

import numpy as np

import oracle
import synth

# relative L2 error bounds per row (token, layer): fp32 1e-5, bf16 1e-2, int4 3e-2
TOL = {"fp32": 1e-5, "bf16": 1e-2, "int4": 3e-2}
NEAR_TIE = 1e-4  # oracle logit gap under which a top-k flip is accepted


def run_gpu(m, hidden: np.ndarray, dtype_out: str):
    """Decode every step of `hidden` [T x L x B x d] through moe_decode_step on device buffers
    (B sequences per step)."""
    import torch

    T = hidden.shape[0]
    dev = torch.device("cuda", 0)
    tdt = torch.float32 if dtype_out == "fp32" else torch.bfloat16
    hid = torch.from_numpy(hidden.view(np.float32) if dtype_out == "fp32" else hidden.view(np.int16))
    hid = hid.to(dev)
    if dtype_out != "fp32":
        hid = hid.view(torch.bfloat16)
    out = torch.empty(hid.shape, dtype=tdt, device=dev)
    idx = np.empty(hidden.shape[:3] + (m.cfg.top_k,), dtype=np.int32)
    gate = np.empty(idx.shape, dtype=np.float32)
    B = hidden.shape[2]
    for t in range(T):
        m.decode_step(hid[t], out[t], batch=B)
        i, g = m.get_last_routing()
        idx[t], gate[t] = i[:, :B], g[:, :B]
    torch.cuda.synchronize()
    o = out.float().cpu().numpy().astype(np.float64)
    return o, idx, gate


def oracle_trace(wl, hidden: np.ndarray, cap: int, forced_idx=None, routers=None, policy="lru"):
    """Routing + residency trace of the oracle for all steps (no expert FFN)."""
    orc = oracle.Oracle.for_workload(wl, cap_slots=cap, keep_slot_copies=False, routers=routers, policy=policy)
    idx, z, recs = [], [], []
    for t in range(hidden.shape[0]):
        r = orc.decode_step(hidden[t], compute_out=False, forced_idx=None if forced_idx is None else forced_idx[t])
        idx.append(r.idx)
        z.append(r.z)
        recs.append(r.records)
    return np.stack(idx), np.stack(z), np.concatenate(recs)


def check_routing(gpu_idx, orc_idx, orc_z, k):
    """Top-k ids must match exactly except swaps among experts whose oracle logits lie within
    NEAR_TIE of the k-th largest. Returns the number of accepted flips."""
    flips = 0
    shp = gpu_idx.shape[:-1]
    for pos in np.ndindex(*shp):
        g, o = gpu_idx[pos], orc_idx[pos]
        if np.array_equal(g, o):
            continue
        z = orc_z[pos]
        zk = np.sort(z)[::-1][k - 1]
        diff = set(g.tolist()) ^ set(o.tolist())
        if not diff:
            # same set, different order: only allowed among near-equal logits
            for a, b in zip(g, o):
                if a != b:
                    assert abs(z[a] - z[b]) < NEAR_TIE, f"rank order differs at {pos}"
            flips += 1
            continue
        for e in diff:
            assert abs(z[e] - zk) < NEAR_TIE, f"top-k set differs at {pos} beyond a near-tie (expert {e})"
        flips += 1
    return flips


def trace_tuples(tr):
    return np.stack([tr["step"], tr["layer"], tr["expert"], tr["kind"], tr["slot"], tr["evicted"]], axis=1)


def rel_l2_rows(gpu_out, ref_out):
    num = np.linalg.norm(gpu_out - ref_out, axis=-1)
    den = np.linalg.norm(ref_out, axis=-1)
    return num / np.maximum(den, 1e-300)
