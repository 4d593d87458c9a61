"""Host-side logic of bench.py: the multi-rank path (two gloo ranks on CPU)
and the JSON line of the reference arm."""
import io
import json
import os
import socket
from contextlib import redirect_stdout

import pytest
import torch.multiprocessing as mp

import bench


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    d = bench.Dist()
    d.init("gloo")
    d.barrier()
    q.put((rank, d.max(float(rank) + 0.5), bench.context_layers(32, rank)))
    d.barrier()
    d.close()


def test_two_gloo_ranks_time_max_and_distinct_contexts():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [1.5, 1.5]          # max over ranks reaches every rank
    a, b = res[0][2], res[1][2]
    assert len(a) == len(b) == 32 and not set(a) & set(b)


def _layer_worker(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    d = bench.Dist()
    d.init("gloo")
    d.barrier()
    mine = bench.context_layers(32, rank, world, "layers")
    # each rank's time is its own layer block's; the job's time is the slowest rank's
    q.put((rank, d.max(1.0 + 0.25 * len(mine) + rank), mine))
    d.barrier()
    d.close()


def test_two_gloo_ranks_split_one_context_by_layer_blocks():
    """The layer-block split of one context over ranks (no data exchange,
    only the barrier and the max of the ranks' times)."""
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_layer_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    a, b = res[0][2], res[1][2]
    assert a == list(range(16)) and b == list(range(16, 32))    # contiguous blocks, one context
    assert res[0][1] == res[1][1] == 1.0 + 0.25 * 16 + 1


def test_layer_blocks_cover_the_context_for_any_rank_count():
    for world in (1, 2, 3, 4, 5, 8):
        blocks = [bench.context_layers(32, r, world, "layers") for r in range(world)]
        assert sum(blocks, []) == list(range(32))
        assert max(map(len, blocks)) - min(map(len, blocks)) <= 1
    assert bench.context_layers(32, 1, 4, "contexts") == list(range(32, 64))


def test_reference_arm_json_line(monkeypatch):
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    buf = io.StringIO()
    with redirect_stdout(buf):
        rc = bench.main(["--impl", "reference", "--workload", "single_head_T1024", "--steps", "1",
                         "--warmup", "0"])
    assert rc == 0
    line = json.loads(buf.getvalue().strip().splitlines()[-1])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in line
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0
    assert "workload" in line["config"]


def test_reference_arm_only_rank0_prints(monkeypatch):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    buf = io.StringIO()
    with redirect_stdout(buf):
        assert bench.main(["--impl", "reference", "--workload", "single_head_T1024"]) == 0
    assert buf.getvalue() == ""


_FAKE_SMI = """#!/bin/bash
# stand-in for nvidia-smi's looped query: one sample every 50 ms, power cap active
while true; do
  printf '%s, 0, 2070, 2070, 612.50, 0x0000000000000004, Not Active, Not Active, Not Active, Active\\n' \\
    "$(date +'%Y/%m/%d %H:%M:%S.%3N')"
  sleep 0.05
done
"""


def test_clock_sampler_keeps_the_samples_of_the_timed_region(monkeypatch, tmp_path):
    import time
    smi = tmp_path / "nvidia-smi"
    smi.write_text(_FAKE_SMI)
    smi.chmod(0o755)
    monkeypatch.setenv("PATH", str(tmp_path) + os.pathsep + os.environ["PATH"])
    c = bench.ClockSampler(0)
    c.start()
    time.sleep(0.4)
    t0 = time.time()
    time.sleep(0.5)
    t1 = time.time()
    time.sleep(0.3)
    clk = c.stop((t0, t1))
    assert clk["in_window"] and clk["sm_mhz"] == 2070.0 and clk["reasons"] == ["sw_power_cap"]
    assert 4 <= clk["samples"] <= 12 < clk["samples_total"]


def test_clock_summary_parsing_and_fallback():
    lines = ["2026/01/02 03:04:05.100, 0, 1980, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active",
             "2026/01/02 03:04:05.300, 0, 2070, 2070, 950.0, 0x4, Not Active, Active, Not Active, Active",
             "2026/01/02 03:04:05.500, 0, [N/A], 2070, 950.0, 0x0, Not Active, Not Active, Not Active, Not Active",
             "garbage"]
    t = bench.ClockSampler._when("2026/01/02 03:04:05.200")
    clk = bench.ClockSampler.parse(lines, (t, t + 0.2))
    assert clk["samples"] == 1 and clk["sm_mhz"] == 2070.0
    assert clk["reasons"] == ["hw_thermal_slowdown", "sw_power_cap"] and clk["samples_total"] == 2
    # no sample inside the window: all samples count, flagged
    clk = bench.ClockSampler.parse(lines, (t + 10, t + 11))
    assert clk["in_window"] is False and clk["samples"] == 2 and clk["sm_mhz"] == 2025.0
    assert bench.ClockSampler.parse(["garbage"]) is None


@pytest.mark.parametrize("layers,heads,k", [(32, 8, 12), (1, 1, 12), (1, 6, 6), (3, 3, 9), (32, 8, 400)])
def test_cpu_baseline_sample_pairs_are_distinct_and_spread(layers, heads, k):
    pairs = bench.cpu_sample_pairs(layers, heads, k)
    assert len(pairs) == len(set(pairs)) == min(k, layers * heads)
    assert all(0 <= l < layers and 0 <= h < heads for l, h in pairs)
    assert pairs[0] == (0, 0) and (k < 2 or layers * heads < 2 or max(l for l, _ in pairs) == layers - 1)


def test_default_timed_steps_follow_the_context_length():
    """About a minute of timed work at 128K (14 steps of ~4.4 s), 20 steps at
    shorter contexts and for the reference arm (whose steps are segments)."""
    assert bench.parse_args([]).steps == 14
    assert bench.parse_args(["--workload", "llama8b_T8192_r10"]).steps == 20
    assert bench.parse_args(["--impl", "reference"]).steps == 20
    assert bench.parse_args(["--steps", "5"]).steps == 5
    assert bench.parse_args([]).warmup >= 3
