"""The bench's `traffic` figure comes from a committed ncu capture of the decode kernel: the capture
must describe the kernel source as it stands (else the bench reports null), and the figure scales
the capture's DRAM bytes per algorithmic byte to the run's own bytes per launch."""
import json
import os

import pytest

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _record():
    with open(os.path.join(ROOT, "profiles", "decode_traffic.json")) as f:
        return json.load(f)


def test_capture_matches_the_decode_kernel_source():
    rec = _record()["ragged"]  # the default workload's capture
    assert rec["kernel_source_hash"] == bench.kernel_source_hash(), \
        "decode kernel changed since profiles/decode_traffic.json was captured: recapture it"


def test_ratio_is_the_captures_own_and_traffic_scales_with_bytes():
    rec = _record()["ragged"]
    cap = rec["captured"]
    ratio = (cap["dram_bytes_read"] + cap["dram_bytes_write"]) / cap["algorithmic_bytes"]
    assert rec["dram_bytes_per_algorithmic_byte"] == pytest.approx(ratio, abs=1e-4)
    assert 0.95 < ratio < 1.05  # each kept row is read once
    assert bench.recorded_traffic("ragged", 1e9) == pytest.approx(ratio * 1e9, rel=1e-3)
    assert bench.recorded_traffic("no-such-workload", 1e9) is None
