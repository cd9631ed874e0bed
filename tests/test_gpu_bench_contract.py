"""bench.py's output line, both arms, on the small workload: one JSON line with
every key and type the benchmark contract names (throughput, roofline of the
dominant kernel, the oracle's CPU baseline, the end-to-end number with its
copied bytes, sampled clocks, the launch count)."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def run(*args):
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT,
                         capture_output=True, text=True, timeout=600, check=True).stdout
    lines = [l for l in out.splitlines() if l.startswith("{")]
    assert len(lines) == 1, out
    return json.loads(lines[0])


def num(x):
    return isinstance(x, (int, float)) and not isinstance(x, bool)


def test_gb300_arm_line():
    d = run("--workload", "tiny", "--steps", "3", "--warmup", "3", "--cpu-seconds", "1")
    for k in ("metric", "unit", "dtype", "data", "scaling"):
        assert isinstance(d[k], str) and d[k]
    assert num(d["value"]) and d["value"] > 0 and num(d["ms_per_step"]) and d["ms_per_step"] > 0
    assert d["n_gpus"] == 1 and d["steps"] == 3 and d["warmup"] == 3
    assert d["higher_is_better"] is True and d["vs_baseline"] is None
    assert d["config"]["workload"] == "tiny"
    r = d["roofline"]
    assert r["bound"] in ("tensor", "hbm", "alu") and r["unit"] in ("TFLOP/s", "GB/s")
    assert num(r["achieved"]) and num(r["peak"]) and r["peak"] > 0
    assert abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-6
    assert r["traffic"] is None or num(r["traffic"])
    c = d["cpu_baseline"]
    assert c["kind"] == "oracle" and num(c["value"]) and c["value"] > 0
    assert isinstance(c["cores"], int) and c["cores"] >= 1 and c["sample"]
    assert c["parity"]["within"] is True and c["parity"]["tokens"] > 0   # the timed outputs
    e = d["e2e"]
    assert num(e["value"]) and e["value"] > 0 and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    assert "sm_mhz" in d["clocks"] and "sm_max_mhz" in d["clocks"]
    assert isinstance(d["clocks"]["reasons"], list)
    assert isinstance(d["gpu_launches"], int) and d["gpu_launches"] >= 3


def test_reference_arm_line():
    d = run("--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "1")
    assert d["impl"] == "reference"
    assert num(d["value"]) and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["value"] == d["value"] and d["e2e"]["unit"] == d["unit"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0


def test_arms_emit_the_same_config():
    """Both arms describe the same workload with the same config keys and
    values, so their lines can be compared directly."""
    a = run("--workload", "tiny", "--steps", "3", "--warmup", "3", "--no-cpu", "--no-e2e")
    b = run("--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "1")
    assert a["config"] == b["config"]
    assert 0 < b["cpu_baseline"]["sample_fraction"] <= 1


def test_graph_replay_line():
    """--graph: the kernel-only steps and the end-to-end steps (input copies,
    the four calls, result copies) are replayed from CUDA graphs; the line
    keeps every key."""
    d = run("--workload", "tiny", "--steps", "3", "--warmup", "3", "--no-cpu", "--graph")
    assert d["config"]["launch"].startswith("CUDA graph")
    e = d["e2e"]
    assert num(e["value"]) and e["value"] > 0 and "graph" in e["overlap"]
    assert e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0


def test_vocab_sharded_line():
    """--shards: re-scoring through hdl_rescore_shard on row shards of W and
    hdl_merge_vocab_shards on one GPU; the timed steps' log-probs still match
    the oracle on its sampled tokens."""
    d = run("--workload", "tiny", "--steps", "3", "--warmup", "3", "--shards", "3",
            "--cpu-seconds", "1", "--no-e2e")
    assert d["config"]["vocab_shards"] == 3
    assert "shards" in d["roofline"]["kernel"] and d["roofline"]["traffic"] is None
    assert d["cpu_baseline"]["parity"]["within"] is True
    assert d["gpu_launches"] == 3 * (2 * 3 + 1 + 3)


def test_entropy_line():
    """--entropy: the re-scoring call also returns the original context's
    next-token entropies (hdl_rescore_ex); both arms report it in config."""
    d = run("--workload", "tiny", "--steps", "3", "--warmup", "3", "--entropy",
            "--cpu-seconds", "1", "--no-e2e")
    assert d["config"]["entropy_orig"] is True and "entropies" in d["roofline"]["kernel"]
    assert d["cpu_baseline"]["parity"]["within"] is True
    b = run("--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "1",
            "--entropy")
    assert b["config"] == d["config"]
