"""Host logic of bench.py on CPU.

The multi-rank path (gloo, world size 2): each GPU runs an independent replica, the job takes as
long as its slowest replica (max over ranks), the job's rate is all replicas' units over that time,
and the reference arm runs on rank 0 only. Also: stored ncu traffic figures are used only for the
kernel sources they were captured on, and the oracle's sample walks units in decode order."""
import os
import socket

import pytest
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, results):
    import torch.distributed as dist

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms_local = [120.0, 95.5][rank]  # rank 0 is the slower replica
        ms = bench.max_over_ranks(ms_local, "cpu")
        rate = bench.whole_job_rate(200 * 64, world, ms * 1e-3)
        dist.barrier()
        results[rank] = (ms, rate)
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_whole_job_rate_on_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as mgr:
        results = mgr.dict()
        port = _free_port()
        procs = [ctx.Process(target=_rank_main, args=(r, 2, port, results)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=120)
        assert all(p.exitcode == 0 for p in procs)
        got = dict(results)
    # both ranks agree on the slowest replica's time and on the job's rate
    assert got[0] == got[1]
    ms, rate = got[0]
    assert ms == 120.0
    assert rate == pytest.approx(2 * 200 * 64 / 0.120)


def test_single_process_needs_no_group():
    assert bench.max_over_ranks(7.5, "cpu") == 7.5
    assert bench.whole_job_rate(10, 1, 2.0) == 5.0


def test_host_tier_guard():
    gb = 1e9
    assert bench.host_tier_fits(60 * gb, 1, int(100 * gb))
    assert not bench.host_tier_fits(60 * gb, 2, int(100 * gb))  # two replicas of a 58 GB tier
    assert bench.host_tier_fits(60 * gb, 8, 0)  # available memory unknown


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    import argparse

    import synth

    monkeypatch.setenv("RANK", "1")
    args = argparse.Namespace(warmup=3, steps=4, gpus=2)
    assert bench.run_reference(args, synth.WORKLOADS["tiny_fp32"]) == 0
    assert capsys.readouterr().out == ""


def test_stored_traffic_only_for_matching_kernel_sources(tmp_path, monkeypatch):
    # a committed ncu summary is used only while the kernel's sources hash to its recorded digest
    prof = tmp_path / "profiles"
    prof.mkdir()
    good = bench.kernel_source_digest("k_fused")
    (prof / "k_ok.md").write_text(f"- kernel_source_digest: `{good}`\n- traffic_bytes_per_full_launch: `12345`\n")
    (prof / "k_stale.md").write_text("- kernel_source_digest: `0000000000000000`\n"
                                     "- traffic_bytes_per_full_launch: `12345`\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "kernel_source_digest", lambda kernel="k_fused": good)
    assert bench.stored_traffic("k_ok.md", "k_fused") == 12345.0
    assert bench.stored_traffic("k_stale.md", "k_fused") is None
    assert bench.stored_traffic("missing.md", "k_fused") is None


def test_sample_units_walk_sequences_then_layers_then_tokens():
    import synth

    wl = synth.WORKLOADS["stack48_batch64"]
    u = bench.sample_units(wl, 130)
    assert u[0] == (0, 0, 0) and u[63] == (0, 0, 63) and u[64] == (0, 1, 0) and u[129] == (0, 2, 1)
    wl1 = synth.WORKLOADS["stack48_bf16"]
    assert bench.sample_units(wl1, 50)[-1] == (1, 1, 0)


def test_decoder_reference_arm_prints_one_line_on_rank_zero(monkeypatch, capsys):
    import argparse
    import json

    import synth

    args = argparse.Namespace(warmup=3, steps=4, gpus=1, impl="reference")
    monkeypatch.setenv("RANK", "1")
    assert bench.run_decoder(args, synth.DECODERS["tiny_block_fp32"]) == 0
    assert capsys.readouterr().out == ""
    monkeypatch.setenv("RANK", "0")
    assert bench.run_decoder(args, synth.DECODERS["tiny_block_fp32"]) == 0
    line = json.loads(capsys.readouterr().out)
    assert line["impl"] == "reference" and line["value"] > 0 and line["cpu_baseline"]["kind"] == "oracle"
    assert line["config"]["workload"] == "tiny_block_fp32"


def test_reference_arm_prints_the_gpu_arms_config(capsys):
    # both arms build `config` from the workload and the options alone, so the driver can compare
    # them key for key; the reference arm's step is one decode token at batch 1
    import json
    from argparse import Namespace

    import synth

    wl = synth.WORKLOADS["tiny_fp32"]
    args = Namespace(gpus=1, steps=2, warmup=3, schedule="device", miss_ctas=0, batched_path="auto", policy="lru",
                     lookahead=True)
    assert bench.run_reference(args, wl) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference"
    assert line["config"] == bench.workload_config(wl, args, 1)
    assert line["config"] == json.loads(json.dumps(bench.workload_config(wl, args, 1)))
    assert line["step"].startswith("one decode token")
    assert line["metric"].startswith("MoE decode tok/s")
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["value"] > 0
