"""Host-side checks of bench.py (no GPU): the reference arm's JSON line and
the hash gate on the ncu traffic figures it quotes."""
from __future__ import annotations

import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

COMPRESS_PROFILE = "compress_kernels_llama3-8b_B4_T32768_8layers.md"
COMPRESS_SOURCES = ["score_tc1.cu", "select.cu", "tc_ptx.cuh", "common.cuh"]


def test_profile_traffic_scales_by_algorithmic_bytes():
    # the committed summary matches the committed sources: its per-launch
    # traffic comes back scaled from the captured launch to the asked one
    fields = {}
    for line in open(os.path.join(ROOT, "profiles", COMPRESS_PROFILE)):
        if ":" in line and not line.startswith(("|", "#", " ")):
            k, v = line.split(":", 1)
            fields[k.strip()] = v.strip()
    traffic = float(fields["traffic_bytes_per_launch"])
    captured = float(fields["algorithmic_bytes_per_launch"])
    got = bench.profile_traffic(COMPRESS_PROFILE, COMPRESS_SOURCES, 2 * captured)
    assert got == round(2 * traffic)


def test_profile_traffic_is_null_once_sources_differ():
    # another source list hashes differently: the figure no longer describes
    # the kernels and is dropped
    assert bench.profile_traffic(COMPRESS_PROFILE, COMPRESS_SOURCES[:1], 1e9) is None
    assert bench.profile_traffic("no_such_summary.md", COMPRESS_SOURCES, 1e9) is None


def test_reference_arm_line():
    # the CPU oracle timed as the reference arm: one JSON line with the
    # contract's keys, the same metric and unit as the GPU arm, and an e2e
    # block that moves nothing between host and device
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "0", "--cpu-seconds", "2"],
                       capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    assert d["n_gpus"] == 1 and d["steps"] == 1 and d["warmup"] == 0
    assert d["higher_is_better"] is True and d["value"] > 0
    assert d["unit"] == "tokens/s"
    assert d["metric"] == bench.METRIC
    cpu = d["cpu_baseline"]
    assert cpu["kind"] == "oracle" and cpu["cores"] >= 1 and cpu["sample"]
    assert cpu["value"] == pytest.approx(d["value"])
    e2e = d["e2e"]
    assert e2e["value"] == pytest.approx(d["value"]) and e2e["unit"] == d["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0
    assert d["config"]["workload"] == "llama3-8b-32L-32q8kv-d128-B4-T32768-bf16"
