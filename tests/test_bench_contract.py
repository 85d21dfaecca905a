"""bench.py's output contract on the host: the reference arm (the oracle
timed on the host cores) prints one JSON line with the keys the driver
reads, and the GPU arm fails loudly, with no JSON line, when there is no
GPU (there is no CPU fallback)."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(*args, timeout=300):
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT,
                          capture_output=True, text=True, timeout=timeout)


def _json_lines(out: str):
    return [json.loads(l) for l in out.splitlines() if l.startswith("{")]


def test_reference_arm_line():
    r = _run("--impl", "reference", "--config", "tiny", "--steps", "2", "--warmup", "3")
    assert r.returncode == 0, r.stderr[-2000:]
    lines = _json_lines(r.stdout)
    assert len(lines) == 1
    d = lines[0]
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference" and d["n_gpus"] == 1 and d["steps"] == 2 and d["warmup"] == 3
    assert d["higher_is_better"] is True and d["value"] > 0 and d["unit"] == "block-tokens/s"
    assert d["config"]["workload"] == "tiny"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"] and cb["value"] == d["value"]
    e2e = d["e2e"]
    assert e2e["value"] == d["value"] and e2e["unit"] == d["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the behaviour without a GPU")
def test_gpu_arm_fails_loudly_without_a_gpu():
    r = _run("--config", "tiny", "--steps", "2", "--warmup", "3", "--no-cpu-baseline")
    assert r.returncode != 0
    assert _json_lines(r.stdout) == []


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_reference_arm_under_torchrun_prints_once():
    # two ranks launched the way the driver launches N > 1: rank 0 alone runs
    # the reference arm and prints; the other rank exits 0 without a line
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "tiny", "--gpus", "2",
           "--steps", "2", "--warmup", "3"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = _json_lines(r.stdout)
    assert len(lines) == 1 and lines[0]["impl"] == "reference" and lines[0]["n_gpus"] == 2


def test_throttled_clock_records_are_taken_again():
    # the rule bench.py applies to its own clock record before it prints
    sys.path.insert(0, ROOT)
    import bench
    ok = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []}
    assert not bench.throttled(ok)
    assert not bench.throttled({"sm_mhz": 1900.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"]})
    for r in ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"):
        assert bench.throttled({"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [r]})
    assert bench.throttled({"sm_mhz": 1200.0, "sm_max_mhz": 2070.0, "reasons": []})   # a clock lock
    assert not bench.throttled({"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]})


def test_mismatch_stats_counts_what_the_arbitration_kept():
    # a hand-built round: K = 3, two sequences
    #   seq 0: drafts [5, 7, 9] vs targets [5, 8, 1]: mismatches at 2 and 3,
    #          position 2 accepted, 3 rejected -> s = 3; one kept, before s
    #   seq 1: drafts [1, 2, 3] vs targets [4, 2, 6]: mismatches at 1 and 3,
    #          both accepted -> s = 4; two kept, both before s
    import types
    sys.path.insert(0, ROOT)
    import bench
    from paper_2605_24793_gb300 import workload as W
    cfg = W.CONFIGS["tiny"].replace(batch=2, k=3)
    rnd = types.SimpleNamespace(
        argmax=torch.tensor([5, 8, 1, 0, 4, 2, 6, 0], dtype=torch.int32),
        draft=torch.tensor([[5, 7, 9], [1, 2, 3]], dtype=torch.int32),
        accept=torch.tensor([[1, 1, 0], [1, 1, 1]], dtype=torch.uint8),
        accept_len=torch.tensor([3, 4], dtype=torch.int32))
    st = bench.mismatch_stats(cfg, rnd)
    assert st == {"mismatch_positions": 4, "mismatches_accepted": 3,
                  "accepted_mismatch_fraction": 0.75, "accepted_mismatches_emitted": 3}
