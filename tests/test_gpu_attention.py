"""The decoder block's attention (moe_attention_decode) through the C ABI against the fp64 oracle's
grouped-query attention on the same inputs: fp32 q, bf16 or fp32 K/V (widened exactly for the
oracle).
Relative L2 error per query head <= 1e-5 (fp32 arithmetic over up to 4096 positions); a single
cached position returns its value row exactly; the kv-head grouping and the split merge are
covered by shapes whose position counts leave ragged splits."""
import numpy as np
import pytest

from oracle.decoder import attend

pytestmark = pytest.mark.gpu

CASES = [  # (n_heads, n_kv_heads, head_dim, max_pos, n_pos)
    (32, 4, 128, 4096, 4095),  # the Qwen3-30B-A3B-class block at context 4096
    (32, 4, 128, 4096, 1000),
    (8, 2, 64, 256, 100),
    (4, 4, 128, 64, 17),
    (16, 2, 128, 512, 333),
    (2, 1, 64, 40, 3),
]


@pytest.fixture(scope="module")
def P():
    import paper_2605_29135_gb300 as P

    P.build()
    return P


def _inputs(Hq, Hkv, D, Tmax, seed, cache="bf16"):
    import torch

    g = torch.Generator().manual_seed(seed)
    cdt = torch.bfloat16 if cache == "bf16" else torch.float32
    q = torch.randn(Hq, D, generator=g, dtype=torch.float32) * 2.0
    K = torch.randn(Hkv, Tmax, D, generator=g, dtype=torch.float32).to(cdt)
    V = torch.randn(Hkv, Tmax, D, generator=g, dtype=torch.float32).to(cdt)
    return q, K, V


@pytest.mark.parametrize("Hq,Hkv,D,Tmax,T", CASES, ids=[f"{c[0]}q{c[1]}kv{c[2]}d_T{c[4]}" for c in CASES])
def test_attention_matches_oracle(P, Hq, Hkv, D, Tmax, T):
    q, K, V = _inputs(Hq, Hkv, D, Tmax, seed=T)
    out = P.attention_decode(q.cuda(), K.cuda(), V.cuda(), T).cpu().numpy().astype(np.float64)
    ref = attend(q.double().numpy(), K.float().double().numpy(), V.float().double().numpy(), T)
    err = np.linalg.norm(out - ref, axis=1) / np.linalg.norm(ref, axis=1)
    assert err.max() <= 1e-5, f"max rel L2 {err.max():.3e}"


@pytest.mark.parametrize("Hq,Hkv,D,Tmax,T", [(4, 2, 64, 40, 33), (8, 1, 128, 600, 599)])
def test_fp32_cache_matches_oracle(P, Hq, Hkv, D, Tmax, T):
    q, K, V = _inputs(Hq, Hkv, D, Tmax, seed=T + 1, cache="fp32")
    out = P.attention_decode(q.cuda(), K.cuda(), V.cuda(), T).cpu().numpy().astype(np.float64)
    ref = attend(q.double().numpy(), K.double().numpy(), V.double().numpy(), T)
    err = np.linalg.norm(out - ref, axis=1) / np.linalg.norm(ref, axis=1)
    assert err.max() <= 1e-5, f"max rel L2 {err.max():.3e}"


def test_single_position_returns_the_value_row(P):
    q, K, V = _inputs(8, 2, 128, 16, seed=5)
    out = P.attention_decode(q.cuda(), K.cuda(), V.cuda(), 1).cpu()
    for h in range(8):
        assert (out[h] == V[h // 4, 0].float()).all()


def test_rejected_arguments(P):
    import torch

    q, K, V = _inputs(8, 2, 128, 16, seed=6)
    with pytest.raises(P.MoEError):
        P.attention_decode(q.cuda(), K.cuda(), V.cuda(), 17)  # past max_pos
    with pytest.raises(P.MoEError):
        P.attention_decode(torch.zeros(12, 128, device="cuda"), K.cuda(), V.cuda(), 4)  # 12 / 2 heads per group
