"""The chained decoder step (moe_decoder_step) through the C ABI against the fp64 decoder oracle
(oracle/decoder.py) on the same seeded weights, KV-cache prefix and token inputs.

- tiny fp32 stack, whole chain: the GPU decodes 8 tokens on its own and every token's output
  stream, every layer's routing and the residency trace match the oracle decoding the same tokens
  (relative L2 <= 1e-5 per row; trace bit-exact; the oracle's k-th / (k+1)-th logit gaps on this
  data are all above 5e-3, so no near-tie can flip a selection);
- full-size bf16 block (d 2048, 32 query / 4 kv heads of 128, 4095 cached positions, E 128, top-8),
  3 layers, and a small int4-expert block (head_dim 64, four query heads per kv head), layer by layer: each piece the GPU logs (attention output, MoE input, MoE output) is
  compared with the oracle applied to the GPU's own input of that piece (teacher forcing), within
  the bf16 tolerance 1e-2; the trace is checked against the oracle's slot group fed the GPU's
  selections (accepted only where they match the oracle's up to near-ties);
- the chain's bookkeeping: the stream entering layer l + 1 is the one entering layer l plus its
  two residual branches, and x_out is the last layer's sum;
- outputs do not depend on the residency cap (bit-identical capped and uncapped);
- errors: a full KV cache, missing layer weights, and handles the decoder cannot drive.
"""
import numpy as np
import pytest

import oracle
import synth
from oracle.decoder import DecoderOracle, rmsnorm
from tests.gpu_harness import TOL, check_routing, rel_l2_rows, trace_tuples

pytestmark = pytest.mark.gpu

TINY = synth.DECODERS["tiny_block_fp32"]
BLOCK3 = synth.DECODERS["block48_bf16"].replace(
    name="block3_bf16", moe=synth.WORKLOADS["stack48_bf16"].replace(n_layers=3, tokens=3, cap_slots=12))
# int4 experts (bf16 attention), head_dim 64, four query heads per kv head, a short cache
SMALL_INT4 = synth.DecoderWorkload(
    "small_int4", synth.Workload("small_int4", d=512, n_experts=16, top_k=4, d_ff=256, n_layers=3, wdtype="int4",
                                 adtype="bf16", tokens=5, batch=1, rho=0.8, cap_slots=10),
    n_heads=8, n_kv_heads=2, head_dim=64, ctx=100)


@pytest.fixture(scope="module")
def P():
    import paper_2605_29135_gb300 as P

    P.build()
    return P


def _run(P, dw, cap_slots=None, tokens=None):
    """Decode `tokens` tokens through the GPU decoder. Returns x_out [T x d] (f64), the layer logs
    [T x L x 4 x d] (f64), the routing [T x L x k] and the residency trace."""
    import torch

    from paper_2605_29135_gb300.workload import create_decoder_for_workload

    T = dw.moe.tokens if tokens is None else tokens
    L, d = dw.moe.n_layers, dw.moe.d
    xs = synth.token_inputs(dw, T)
    m, dec = create_decoder_for_workload(dw, cap_slots=cap_slots, max_tokens=T)
    try:
        tdt = torch.float32 if dw.moe.adtype == "fp32" else torch.bfloat16
        x_in = torch.from_numpy(xs.view(np.float32) if dw.moe.adtype == "fp32" else xs.view(np.int16)).cuda()
        x_in = x_in.view(tdt)
        x_out = torch.empty((T, d), dtype=torch.float32, device="cuda")
        log = torch.empty((T, L, 4, d), dtype=torch.float32, device="cuda")
        idx = np.empty((T, L, dw.moe.top_k), dtype=np.int32)
        for t in range(T):
            assert dec.position == dw.ctx + t
            dec.step(x_in[t], x_out[t], log[t])
            i, _ = m.get_last_routing()
            idx[t] = i[:, 0]
        torch.cuda.synchronize()
        tr = m.get_residency_trace()
    finally:
        dec.destroy()
        m.destroy()
    return x_out.cpu().numpy().astype(np.float64), log.cpu().numpy().astype(np.float64), idx, tr


def test_tiny_fp32_chain_matches_the_oracle(P):
    dw = TINY
    out, log, idx, tr = _run(P, dw)
    orc = DecoderOracle(dw)
    xs = synth.token_inputs(dw)
    ref, ref_idx, recs = [], [], []
    for t in range(xs.shape[0]):
        r = orc.decode_token(synth.act_to_f64(xs[t], dw.moe.adtype))
        ref.append(r.out)
        ref_idx.append(r.idx)
        recs.append(r.records)
        for l in range(dw.moe.n_layers):
            assert rel_l2_rows(log[t, l, 1], r.attn[l]) <= TOL["fp32"], (t, l, "attention")
            assert rel_l2_rows(log[t, l, 2], r.moe_in[l]) <= TOL["fp32"], (t, l, "MoE input")
            assert rel_l2_rows(log[t, l, 3], r.moe_out[l]) <= TOL["fp32"], (t, l, "MoE output")
    assert np.array_equal(idx, np.stack(ref_idx))
    assert np.array_equal(trace_tuples(tr), trace_tuples(np.concatenate(recs)))
    err = rel_l2_rows(out, np.stack(ref))
    assert err.max() <= TOL["fp32"], f"max rel L2 {err.max():.3e}"


def _teacher_forced(dw, log, idx):
    """Apply the oracle to the GPU's own inputs of each piece; returns the largest relative errors
    (attention, MoE input, MoE output) and the oracle's residency records fed the GPU's
    selections."""
    orc = DecoderOracle(dw)
    moe = orc.moe
    T, L = log.shape[0], log.shape[1]
    worst = np.zeros(3)
    recs = []
    for t in range(T):
        for l in range(L):
            x = log[t, l, 0]
            attn = orc.attention(l, x)
            worst[0] = max(worst[0], rel_l2_rows(log[t, l, 1], attn))
            m_ref = rmsnorm(x + log[t, l, 1], orc.attn_w[l]["norm_post"], dw.eps)
            worst[1] = max(worst[1], rel_l2_rows(log[t, l, 2], m_ref))
            # the MoE layer on the GPU's stored input: routing up to near-ties, then the oracle's
            # slot group and experts fed the GPU's selection
            m_gpu = log[t, l, 2][None, :]
            oi, _, oz, _ = oracle.router(moe.routers[l], m_gpu[0], moe.k, moe.renorm)
            check_routing(idx[t, l][None, :], oi[None, :], oz[None, :], moe.k)
            o, _, _, _, r = moe.layer_step(l, m_gpu, forced_idx=[idx[t, l]])
            worst[2] = max(worst[2], rel_l2_rows(log[t, l, 3], o[0]))
            recs.append(r)
        moe.token_step += 1
        orc.pos += 1
    return worst, np.concatenate(recs)


def test_bf16_block_layer_by_layer_matches_the_oracle(P):
    dw = BLOCK3
    out, log, idx, tr = _run(P, dw)
    worst, recs = _teacher_forced(dw, log, idx)
    assert worst.max() <= TOL["bf16"], f"attention / MoE input / MoE output rel L2 {worst}"
    assert np.array_equal(trace_tuples(tr), trace_tuples(recs))
    _check_chain(out, log)


def test_int4_block_layer_by_layer_matches_the_oracle(P):
    dw = SMALL_INT4
    out, log, idx, tr = _run(P, dw)
    worst, recs = _teacher_forced(dw, log, idx)
    assert worst[:2].max() <= TOL["bf16"] and worst[2] <= TOL["int4"], f"rel L2 {worst}"
    assert np.array_equal(trace_tuples(tr), trace_tuples(recs))
    assert (tr["evicted"] >= 0).any()
    _check_chain(out, log)


def test_block48_bf16_full_size_sampled_layers(P):
    # the bench's workload (48 blocks, 4095 cached positions, 6 GB pool): the trace of every layer
    # against the oracle's slot group fed the GPU's selections, the pieces of sampled layers against
    # the oracle on the GPU's own inputs
    dw = synth.DECODERS["block48_bf16"]
    T, sampled = 2, (0, 23, 47)
    out, log, idx, tr = _run(P, dw, tokens=T)
    moe = oracle.Oracle.for_workload(dw.moe, keep_slot_copies=False)
    orc = DecoderOracle(dw, layers=sampled, max_tokens=T, moe=moe)
    worst, recs = np.zeros(3), []
    for t in range(T):
        for l in range(dw.moe.n_layers):
            m_gpu = log[t, l, 2][None, :]
            oi, _, oz, _ = oracle.router(moe.routers[l], m_gpu[0], moe.k, moe.renorm)
            check_routing(idx[t, l][None, :], oi[None, :], oz[None, :], moe.k)
            o, _, _, _, r = moe.layer_step(l, m_gpu, compute_out=l in sampled, forced_idx=[idx[t, l]])
            recs.append(r)
            if l in sampled:
                x = log[t, l, 0]
                worst[0] = max(worst[0], rel_l2_rows(log[t, l, 1], orc.attention(l, x)))
                m_ref = rmsnorm(x + log[t, l, 1], orc.attn_w[l]["norm_post"], dw.eps)
                worst[1] = max(worst[1], rel_l2_rows(log[t, l, 2], m_ref))
                worst[2] = max(worst[2], rel_l2_rows(log[t, l, 3], o[0]))
        moe.token_step += 1
        orc.pos += 1
    assert worst.max() <= TOL["bf16"], f"attention / MoE input / MoE output rel L2 {worst}"
    assert np.array_equal(trace_tuples(tr), trace_tuples(np.concatenate(recs)))
    _check_chain(out, log)


def _check_chain(out, log):
    T, L = log.shape[0], log.shape[1]
    for t in range(T):
        for l in range(L):
            nxt = out[t] if l == L - 1 else log[t, l + 1, 0]
            want = log[t, l, 0] + log[t, l, 1] + log[t, l, 3]
            assert rel_l2_rows(nxt, want) <= 1e-6, (t, l)


def test_tiny_fp32_chain_bookkeeping(P):
    out, log, _, _ = _run(P, TINY, tokens=3)
    _check_chain(out, log)
    assert np.array_equal(log[:, 0, 0], synth.act_to_f64(synth.token_inputs(TINY, 3), "fp32"))


def test_outputs_do_not_depend_on_the_cap(P):
    dw = TINY
    capped, log_c, idx_c, tr_c = _run(P, dw, cap_slots=dw.moe.top_k * 2, tokens=6)
    full, log_f, idx_f, tr_f = _run(P, dw, cap_slots=dw.moe.n_layers * dw.moe.n_experts, tokens=6)
    assert (tr_c["kind"] == 1).sum() > (tr_f["kind"] == 1).sum()  # the cap did evict
    assert np.array_equal(idx_c, idx_f)
    assert np.array_equal(capped, full) and np.array_equal(log_c, log_f)


def test_full_cache_missing_weights_and_unsupported_handles(P):
    import torch

    from paper_2605_29135_gb300.workload import create_decoder_for_workload, create_for_workload

    dw = TINY
    m, dec = create_decoder_for_workload(dw, max_tokens=1)
    try:
        x = torch.zeros(dw.moe.d, dtype=torch.float32, device="cuda")
        y = torch.empty(dw.moe.d, dtype=torch.float32, device="cuda")
        dec.step(x, y)
        with pytest.raises(P.MoEError) as ei:
            dec.step(x, y)
        assert ei.value.status == -4 and "full" in str(ei.value)
        assert dec.position == dw.ctx + 1
        dec.set_cache(0, *synth.kv_prefix(dw, 0))  # layer 0 now holds ctx positions, layer 1 ctx + 1
        with pytest.raises(P.MoEError) as ei:
            dec.step(x, y)
        assert ei.value.status == -1
    finally:
        dec.destroy()
        m.destroy()
    m = create_for_workload(dw.moe)
    try:
        dec = P.Decoder(m, dw.n_heads, dw.n_kv_heads, dw.head_dim, max_pos=dw.ctx + 4)
        try:
            with pytest.raises(P.MoEError) as ei:
                dec.step(torch.zeros(dw.moe.d, device="cuda"), torch.empty(dw.moe.d, device="cuda"))
            assert ei.value.status == -5
        finally:
            dec.destroy()
        with pytest.raises(P.MoEError):
            P.Decoder(m, dw.n_heads, dw.n_kv_heads, 96, max_pos=8)  # head_dim 96
    finally:
        m.destroy()
    m = create_for_workload(dw.moe, schedule="host_copy_engine")
    try:
        with pytest.raises(P.MoEError) as ei:
            P.Decoder(m, dw.n_heads, dw.n_kv_heads, dw.head_dim, max_pos=8)
        assert "device schedule" in str(ei.value)
    finally:
        m.destroy()


def test_a_moe_layer_that_times_out_is_reported_by_the_next_step_and_the_decoder_recovers(P):
    # an injected barrier fault makes the first MoE launch's waits run out (0.2 s); the device flag
    # is sticky, so the step's later MoE launches leave at once. The next decoder step reports
    # MOE_ERR_TIMEOUT before doing any MoE work, leaves the position where it was, and the steps
    # after it run on an emptied pool
    import torch

    from paper_2605_29135_gb300.workload import create_decoder_for_workload

    dw = TINY
    xs = torch.from_numpy(synth.token_inputs(dw, 4).view(np.float32)).cuda()
    y = torch.empty(dw.moe.d, dtype=torch.float32, device="cuda")
    m, dec = create_decoder_for_workload(dw, max_tokens=4)
    try:
        dec.step(xs[0], y)
        m.inject_fault("barrier_timeout")
        dec.step(xs[1], y)
        torch.cuda.synchronize()
        pos = dec.position
        with pytest.raises(P.MoEError) as ei:
            dec.step(xs[2], y)
        assert ei.value.status == -6 and dec.position == pos
        dec.step(xs[2], y)
        torch.cuda.synchronize()
        assert np.isfinite(y.cpu().numpy()).all()
        tr = m.get_residency_trace()
        assert tr["step"].max() == 0 and (tr["kind"] == 1).all()  # a cold pool again, step 0
    finally:
        dec.destroy()
        m.destroy()
