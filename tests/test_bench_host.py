"""Host-side pieces of bench.py that need no GPU: the algorithmic FLOP count
of a block and the clock sampler's summary of nvidia-smi samples (driven by
a stand-in nvidia-smi on PATH that prints fixed samples)."""
import os
import stat
import sys
import time

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2606_13898_gb300 import inputs as I  # noqa: E402


def test_block_flops_counts_gemms_and_joint_attention():
    wl = I.block_64(keep_ratio="1/4")
    d, T = wl.d, wl.T
    rows = 1877
    M = T + rows
    assert bench.block_flops(wl, [0, rows]) == 24.0 * M * d * d + 4.0 * M * M * d
    # attention-only layer: QKV and out-projection only (8 M d^2)
    tl = I.tiny_layer()
    assert bench.block_flops(tl, [0, 100]) == 8.0 * (tl.T + 100) * tl.d ** 2 + 4.0 * (tl.T + 100) ** 2 * tl.d


FAKE = """#!/bin/sh
while true; do
  echo "0, 1990, 2070, 950.0, 0x4, Not Active, Not Active, Not Active, Active"
  echo "0, 2010, 2070, 960.0, 0x0, Not Active, Active, Not Active, Not Active"
  echo "garbage line"
  sleep 0.05
done
"""


def test_clock_sampler_summarises_samples(tmp_path, monkeypatch):
    smi = tmp_path / "nvidia-smi"
    smi.write_text(FAKE)
    smi.chmod(smi.stat().st_mode | stat.S_IEXEC)
    monkeypatch.setenv("PATH", f"{tmp_path}{os.pathsep}{os.environ['PATH']}")
    c = bench.ClockSampler(0)
    c.start()
    time.sleep(0.5)
    got = c.stop()
    assert got is not None and got["samples"] >= 4
    assert 1990.0 <= got["sm_mhz"] <= 2010.0 and got["sm_max_mhz"] == 2070.0
    assert got["reasons"] == ["hw_thermal_slowdown", "sw_power_cap"]


def test_clock_sampler_without_nvidia_smi(monkeypatch, tmp_path):
    monkeypatch.setenv("PATH", str(tmp_path))  # an empty directory: no nvidia-smi
    c = bench.ClockSampler(0)
    c.start()
    assert c.stop() is None


def test_reference_arm_reports_the_gpu_arms_config(monkeypatch, capsys):
    # The reference arm (the oracle on the host) must describe the same
    # workload as the GPU arm: identical config keys and values, including
    # the packed row count of the workload's split. The oracle's steps are
    # stubbed out here; only the line is checked.
    import json
    monkeypatch.setattr(bench, "oracle_step", lambda sample: None)
    monkeypatch.setattr(bench, "oracle_sample", lambda ratio, crop, seed_offset=0: (None, I.make_batch(
        I.tiny_layer()).x, None, None, None, None, None, 8))
    for v in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(v, raising=False)
    bench.run_reference(bench.parse(["--impl", "reference", "--steps", "1", "--warmup", "0"]))
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference"
    wl = bench.workload("1/4")
    gpu_cfg = bench.line_config(wl, "1/4", line["config"]["packed_image_rows"], 1)
    assert line["config"] == gpu_cfg
    assert line["config"]["packed_image_rows"] == 1877 and line["config"]["block_rows"] == 2389


def test_oracle_config_baseline_single_and_multi_block():
    # The per-configuration oracle timing runs the oracle's own hot path: a
    # single block in one pass, and a stack of blocks one timed step at a
    # time (extrapolated to 28 steps). Tiny 32x32 layers keep it quick.
    wl = I.tiny_layer()
    b = I.make_batch(wl)
    ws = [I.make_weights(wl.d, wl.mlp, seed=I.weight_seed(wl, i)) for i in range(2)]
    one = bench.oracle_config_baseline(wl, b, ws[:1])
    assert one["kind"] == "oracle" and one["value"] > 0 and one["cores"] >= 1
    two = bench.oracle_config_baseline(wl, b, ws)
    assert two["value"] > 0
    assert two["seconds_28_steps_extrapolated"] == 28 * two["seconds_per_step"]
