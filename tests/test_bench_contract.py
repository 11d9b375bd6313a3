"""The reference arm of bench.py (the fp64 oracle on the host cores) prints one
JSON line with the keys the benchmark contract asks for; it needs no GPU, so
the line is checked here on a small workload."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(*args):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    return json.loads(lines[0])


def test_reference_arm_line():
    d = _run("--impl", "reference", "--workload", "tiny_f32", "--steps", "2", "--warmup", "1")
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "impl", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["value"] > 0 and d["unit"] == "tokens/s"
    assert d["n_gpus"] == 1 and d["steps"] == 2 and d["warmup"] == 1 and d["higher_is_better"] is True
    assert d["data"] == "synthetic" and d["dtype"] == "f64" and d["vs_baseline"] is None
    assert "tiny_f32" in d["config"]["workload"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    e2e = d["e2e"]
    assert e2e["value"] == d["value"] and e2e["unit"] == d["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0


def test_reference_arm_decode():
    """The decode workload's reference arm: the oracle recomputes each sampled head's causal
    output over the prefill and the new token (it keeps no state)."""
    d = _run("--impl", "reference", "--workload", "decode", "--steps", "1", "--warmup", "0")
    assert d["impl"] == "reference" and d["value"] > 0 and d["unit"] == "tokens/s" and "decode" in d["metric"]
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and "prefill of n=1024" in d["config"]["workload"]


def test_channel_rms_option():
    """--ch-rms-target runs the normalised feature map and names it in the workload;
    the decode workload rejects it before any work."""
    d = _run("--impl", "reference", "--workload", "tiny_f32", "--steps", "1", "--warmup", "0", "--ch-rms-target",
             "0.1")
    assert d["value"] > 0 and "channel RMS normalisation target 0.1" in d["config"]["workload"]
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--workload", "decode", "--ch-rms-target",
                        "0.1"], cwd=ROOT, capture_output=True, text=True, timeout=120)
    assert r.returncode == 2 and "decode step" in r.stderr


def test_algorithmic_bytes_by_hand():
    """Per-launch algorithmic bytes on a small non-causal case worked out by hand:
    B = 2, H = 1, n = 256, d = dv = 32, D = 64, bf16, lengths (256, 100):
    valid rows 356, all rows 512, statistics 2 x (64*32 + 64) x 4 B = 16896 B."""
    sys.path.insert(0, ROOT)
    import dataclasses
    import numpy as np
    import bench
    from synth.workloads import WORKLOADS
    w = dataclasses.replace(WORKLOADS["lra"], B=2, H=1, n=256)
    ln = np.array([256, 100], dtype=np.int32)
    row = 32 * 2  # one row of Q, K, V or their gradients in bf16
    assert bench.kernel_bytes(w, ln, "tc_keys") == 356 * 2 * row + 16896
    assert bench.kernel_bytes(w, ln, "tc_query") == 356 * row + 512 * row + 16896
    assert bench.kernel_bytes(w, ln, "tc_bwd_query") == 356 * 2 * row + 512 * row + 2 * 16896
    assert bench.kernel_bytes(w, ln, "tc_bwd_key") == 356 * 2 * row + 512 * 2 * row + 16896
    assert bench.kernel_bytes(w, ln, "chrms_stats") == bench.kernel_bytes(w, ln, "tc_chstats") == 2 * 356 * row
    assert bench.kernel_bytes(w, ln, "tc_kterm") == bench.kernel_bytes(w, ln, "chrms_kterm")
    assert bench.kernel_bytes(w, ln, "chrms_kterm") == 2 * 356 * 3 * row
    assert bench.kernel_bytes(w, ln, "no_such_kernel") == 0.0


def test_streaming_form_algorithmic_bytes_by_hand():
    """The streaming-form stages count only the method's tensors they read or write:
    B = 1, H = 2, n = 300, d = dv = 128, bf16 (a row is 256 B), no padding: 600 rows.
    The stage that reads only another stage's rows has no algorithmic bytes."""
    sys.path.insert(0, ROOT)
    import dataclasses
    import bench
    from synth.workloads import WORKLOADS
    w = dataclasses.replace(WORKLOADS["causal_long"], B=1, H=2, n=300)
    row = 128 * 2
    assert bench.kernel_bytes(w, None, "tc_causal") == 600 * 3 * row + 600 * row  # Q, K, V; O
    assert bench.kernel_bytes(w, None, "tc_keys") == 600 * 2 * row                 # K, V
    assert bench.kernel_bytes(w, None, "tcc_query") == 600 * 4 * row               # Q, K, V, dO
    assert bench.kernel_bytes(w, None, "tcc_dstats") == 0.0
    assert bench.kernel_bytes(w, None, "tcc_key") == 600 * 2 * row + 600 * row     # V, dO; dV
    assert bench.kernel_bytes(w, None, "tc_phi_bwd") == 600 * row + 600 * row      # X; dX
    # the whole step: read Q, K, V and write O; read Q, K, V, dO and write dQ, dK, dV
    assert bench.step_bytes(w, None) == 600 * row * (4 + 7)


def test_reference_arm_streaming_form_sample_is_bounded_and_labelled():
    """The streaming-form workload's reference arm times a prefix sample of each sequence and says that its
    per-step time is extrapolated from the sample's rate."""
    d = _run("--impl", "reference", "--workload", "causal_long", "--steps", "1", "--warmup", "0")
    assert d["impl"] == "reference" and d["value"] > 0
    assert "first 4096" in d["cpu_baseline"]["sample"]
    assert d["ms_per_step_kind"].startswith("extrapolated")
    assert d["sample_seconds_per_step"] < 60
