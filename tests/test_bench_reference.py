"""The reference arm of bench.py (the fp64 oracle on the host cores): its JSON line carries every
key of the bench contract, and under a multi-rank launch only rank 0 runs and prints."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(extra_env, gpus):
    env = dict(os.environ, **extra_env)
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
           "--steps", "2", "--warmup", "1", "--gpus", str(gpus)]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    return [json.loads(l) for l in r.stdout.splitlines() if l.startswith("{")]


def _check_line(line, gpus):
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in line, k
    assert line["impl"] == "reference" and line["n_gpus"] == gpus
    assert line["steps"] == 2 and line["warmup"] == 1 and line["higher_is_better"] is True
    assert line["value"] > 0 and line["ms_per_step"] > 0 and line["vs_baseline"] is None
    assert line["config"]["workload"].startswith("tiny")
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == line["value"] and cb["sample"]
    e = line["e2e"]
    assert e["value"] == line["value"] and e["unit"] == line["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0
    # tiny's one layer is timed whole every step: the step time is what ran, and the value follows from it
    assert line["extrapolated"] is False and line["layers_timed_per_step"] == 1
    assert abs(line["value"] - 2 / (line["ms_per_step"] / 1e3)) <= 1e-9 * line["value"]


def test_reference_arm_times_every_layer_where_the_history_fits():
    """The OPT-1.3B-shaped history (~7 GB of K/V) is timed layer by layer in full; the ragged one
    (~100 GB) is sampled at layer 0 and flagged as extrapolated."""
    sys.path.insert(0, ROOT)
    import bench
    from synth import workloads as wl

    layers, nbytes = bench.reference_layers(wl.opt13b(), 25)
    assert layers == list(range(24)) and nbytes < bench.REFERENCE_ALL_LAYERS_BYTES
    layers, nbytes = bench.reference_layers(wl.ragged(), 25)
    assert layers == [0] and nbytes > 50e9


def test_reference_arm_single_rank():
    lines = _run({"RANK": "0", "WORLD_SIZE": "1", "LOCAL_RANK": "0"}, 1)
    assert len(lines) == 1
    _check_line(lines[0], 1)


def test_reference_arm_two_ranks_only_rank0_prints():
    assert _run({"RANK": "1", "WORLD_SIZE": "2", "LOCAL_RANK": "1"}, 2) == []
    lines = _run({"RANK": "0", "WORLD_SIZE": "2", "LOCAL_RANK": "0"}, 2)
    assert len(lines) == 1
    _check_line(lines[0], 2)
