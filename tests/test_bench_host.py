"""Host logic of bench.py: max-over-ranks timing and whole-job throughput on two gloo ranks (CPU)."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = 10.0 + 5.0 * rank                # the slower rank sets the job time
        got = bench.max_over_ranks(ms)
        out[rank] = got
        out[world + rank] = bench.job_throughput(100.0, 4, world, got)
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_throughput_gloo():
    world = 2
    out = mp.get_context("spawn").Manager().list([0.0] * (2 * world))
    mp.start_processes(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True,
                       start_method="spawn")
    assert list(out[:world]) == [15.0, 15.0]
    # 2 ranks x 100 units x 4 steps in 15 ms
    assert out[world] == pytest.approx(2 * 100 * 4 / 0.015)
    assert out[world] == out[world + 1]


def test_single_process_defaults():
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.job_throughput(65536, 20, 1, 1000.0) == pytest.approx(65536 * 20)


def test_reference_arm_nonzero_rank_does_no_work(monkeypatch):
    monkeypatch.setenv("RANK", "1")
    args = type("A", (), {"workload": "7b-16k-w4", "ref_rows": 8, "steps": 1, "warmup": 0,
                          "gpus": 2})()
    assert bench.run_reference(args) == 0


def test_algorithmic_work_7b_matches_hand_count():
    import synth
    wl = synth.workload("7b-16k-w4")
    flops, byts = bench.algorithmic_work(wl.model, wl.lora, 16384)
    # base GEMMs: 2 * n * sum(in * out) over the seven projections
    h, f, qd, kvd = 3584, 18944, 3584, 512
    base = 2 * 16384 * (h * (qd + 2 * kvd) + qd * h + 2 * h * f + f * h)
    gemm = sum(v for k, v in flops.items() if k.startswith("gemm_"))
    # adapter: down products over each module's input, up products over its output
    lora_up = 2 * 16384 * 16 * (qd + 2 * kvd + h + 2 * f + h)
    lora_down = 2 * 16384 * 16 * (3 * h + qd + 2 * h + f)
    assert gemm == base + lora_up + lora_down
    assert flops["attn_prefill_paged"] == 4 * 28 * 128 * 16384 * 16385 // 2


def test_shard_requests_partitions_and_balances():
    import synth
    wl = synth.workload("7b-batch8")
    loads = [(e - s) * n for n, (s, e) in zip(wl.n_tokens, wl.windows)]
    for world in (1, 2, 4, 8):
        parts = bench.shard_requests(loads, world)
        flat = sorted(i for p in parts for i in p)
        assert flat == list(range(len(loads)))          # every request exactly once
        tot = [sum(loads[i] for i in p) for p in parts]
        assert max(tot) - min(tot) <= max(loads)        # greedy LPT balance bound
    assert bench.shard_requests([7], 3) == [[0], [0], [0]]   # one prefix: replicas


def test_reference_arm_line_has_the_contract_keys(capsys, monkeypatch):
    """The reference arm (the oracle on the host cores) prints one JSON line with the metric,
    its own cpu_baseline and an e2e object that copies nothing between host and device."""
    import json
    monkeypatch.delenv("RANK", raising=False)
    args = type("A", (), {"workload": "tiny", "ref_rows": 16, "steps": 1, "warmup": 0, "gpus": 1,
                          "lora_rank": 0, "lora_modules": ""})()
    assert bench.run_reference(args) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    for key in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC and line["unit"] == bench.UNIT
    assert line["higher_is_better"] is True and line["value"] > 0
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == line["value"] and cb["cores"] >= 1 and cb["sample"]
    e2e = line["e2e"]
    assert e2e["value"] == line["value"] and e2e["unit"] == line["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0
    assert "tiny" in line["config"]["workload"] and "tiny" in line["data"]


def test_clock_summary_reports_median_and_active_reasons():
    rows = ["0, 1950, 2070, 900.1, 0x4, Not Active, Not Active, Not Active, Active\n",
            "0, 1980, 2070, 1200.5, 0x0, Not Active, Not Active, Not Active, Not Active\n",
            "0, 1400, 2070, 1390.0, 0x4, Not Active, Not Active, Not Active, Active\n",
            "garbage line\n"]
    s = bench.ClockSampler.summarise(rows)
    assert s["sm_mhz"] == 1950.0 and s["sm_max_mhz"] == 2070.0 and s["samples"] == 3
    assert s["reasons"] == ["sw_power_cap"]
    hot = bench.ClockSampler.summarise(["0, 1500, 2070, 1000, 0x40, Not Active, Active, Not Active, Not Active\n"])
    assert hot["reasons"] == ["hw_thermal_slowdown"]
    assert bench.ClockSampler.summarise([])["reasons"] == ["no samples"]
    na = bench.ClockSampler.summarise(["0, [N/A], [N/A], [N/A], [N/A], [N/A], [N/A], [N/A], [N/A]\n"])
    assert na["sm_mhz"] is None and na["sm_max_mhz"] is None


def test_step_bytes_7b_match_hand_count():
    import synth
    wl = synth.workload("7b-16k-w4")
    b = bench.step_bytes(wl.model, wl.lora, wl.n_tokens, wl.windows)
    h, f, qd, kvd, r, N = 3584, 18944, 3584, 512, 16, 28
    per_layer_w = 2 * (h * (qd + 2 * kvd) + qd * h + 2 * h * f + f * h)
    per_layer_lora = 2 * r * ((h + qd) + 2 * (h + kvd) + (qd + h) + 2 * (h + f) + (f + h))
    assert b["drift_gram"] == 2 * N * per_layer_lora == 161480704
    # window [14, 18): the row runs layers 18..27 over 16383 cached keys per layer (K and V)
    assert b["tail_decode"] == 10 * (per_layer_w + per_layer_lora + 2 * 16383 * kvd * 2)
    assert b["lm_head"] == 152064 * h * 2
