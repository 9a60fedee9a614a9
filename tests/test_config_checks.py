"""The boundary's configuration checks, on CPU: moe_create validates a configuration before it
touches a device, so every invalid field is reported as MOE_ERR_INVALID with a message naming the
problem; moe_expert_bytes / moe_pool_bytes answer for valid configurations and return -1 for
invalid ones."""
import pytest

import paper_2605_29135_gb300 as P
from paper_2605_29135_gb300.buildsys import build

BASE = dict(d=256, n_experts=8, top_k=2, d_ff=128, n_layers=1, wdtype="fp32", adtype="fp32", cap_slots=4)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build()


def _cfg(**over):
    args = dict(BASE)
    raw = {k: over.pop(k) for k in list(over) if k.startswith("raw_")}
    args.update(over)
    cfg = P.make_config(args.pop("d"), args.pop("n_experts"), args.pop("top_k"), args.pop("d_ff"),
                        args.pop("n_layers"), args.pop("wdtype"), args.pop("adtype"), **args)
    for k, v in raw.items():  # fields set past the Python helper's checks
        setattr(cfg, k[4:], v)
    return cfg


BAD = [
    (dict(d=0), "must be positive"),
    (dict(n_experts=257), "n_experts must be <= 256"),
    (dict(top_k=17, n_experts=32), "top_k must be <= 16"),
    (dict(top_k=9), "<= n_experts"),
    (dict(max_batch=0), "max_batch must be in [1, 64]"),
    (dict(max_batch=65), "max_batch must be in [1, 64]"),
    (dict(max_batch=2, schedule="host_copy_engine"), "needs the device schedule"),
    (dict(adtype="bf16"), "fp32 weights need fp32 activations"),
    (dict(d=258), "multiples of 4"),
    (dict(d=4096), "fp32 needs d <= 2048"),
    (dict(wdtype="bf16", adtype="bf16", d_ff=132), "multiples of 8"),
    (dict(wdtype="bf16", adtype="bf16", d=8192), "bf16 needs d <= 4096"),
    (dict(wdtype="int4", adtype="bf16", d=384, d_ff=100), "multiples of 128"),
    (dict(wdtype="int4", adtype="fp32"), "int4 weights need bf16 activations"),
    (dict(raw_wdtype=7), "unknown wdtype"),
    (dict(wdtype="bf16", adtype="bf16", d_ff=4104), "d_ff too large"),
    (dict(wdtype="bf16", adtype="bf16", top_k=8, d_ff=4096, d=1024), "too large"),
    (dict(raw_renorm=2), "renorm must be 0 or 1"),
    (dict(trace_capacity=-1), "trace_capacity must be >= 0"),
    (dict(raw_schedule=5), "unknown schedule"),
    (dict(miss_ctas=-1), "miss_ctas must be >= 0"),
    (dict(raw_batched_path=3), "unknown batched_path"),
    (dict(raw_policy=9), "unknown policy"),
    (dict(policy="rotary", max_batch=4, schedule="host_copy_engine"), "max_batch above 1 needs the device schedule"),
    (dict(raw_lookahead=2), "lookahead must be 0 or 1"),
    (dict(lookahead=True, max_batch=4), "lookahead in the device schedule needs max_batch 1 and the LRU policy"),
    (dict(lookahead=True, policy="rotary"), "lookahead in the device schedule needs max_batch 1 and the LRU policy"),
]


@pytest.mark.parametrize("over,msg", BAD, ids=[m for _, m in BAD])
def test_invalid_configuration_is_rejected_before_any_device_work(over, msg):
    cfg = _cfg(**over)
    with pytest.raises(P.MoEError) as ei:
        P.MoE(cfg)
    assert ei.value.status == -1
    assert msg in str(ei.value)
    lib = P._lib.load()
    import ctypes

    assert lib.moe_expert_bytes(ctypes.byref(cfg)) == -1
    assert lib.moe_pool_bytes(ctypes.byref(cfg)) == -1


@pytest.mark.parametrize("wdtype,adtype,d,I,expect", [
    ("fp32", "fp32", 256, 128, 3 * 256 * 128 * 4),
    ("bf16", "bf16", 2048, 768, 9437184),
    ("int4", "bf16", 2048, 768, 3 * 2048 * 768 // 2 + 3 * 2048 * 768 // 128 * 2),
])
def test_expert_and_pool_bytes(wdtype, adtype, d, I, expect):
    import ctypes

    lib = P._lib.load()
    cfg = _cfg(wdtype=wdtype, adtype=adtype, d=d, d_ff=I, cap_slots=10, n_layers=3)
    eb = lib.moe_expert_bytes(ctypes.byref(cfg))
    assert eb == expect
    stride = (eb + 255) // 256 * 256
    assert lib.moe_pool_bytes(ctypes.byref(cfg)) == 10 * stride
    # a cap above the stack's expert count is clipped to it; a byte budget gives whole slots
    cfg = _cfg(wdtype=wdtype, adtype=adtype, d=d, d_ff=I, cap_slots=1000, n_layers=3)
    assert lib.moe_pool_bytes(ctypes.byref(cfg)) == 3 * 8 * stride
    cfg = _cfg(wdtype=wdtype, adtype=adtype, d=d, d_ff=I, cap_slots=0, cap_bytes=5 * stride + 7, n_layers=3)
    assert lib.moe_pool_bytes(ctypes.byref(cfg)) == 5 * stride
