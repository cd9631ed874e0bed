"""The reference arm of bench.py (the fp64 oracle timed on the host cores)
on CPU: one JSON line with the contract's keys; under torchrun with two
ranks only rank 0 prints it and every rank exits 0."""
import json
import os
import socket
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def json_lines(out: str):
    return [json.loads(l) for l in out.splitlines() if l.startswith("{")]


def env():
    e = dict(os.environ)
    e["CUDA_VISIBLE_DEVICES"] = ""
    return e


def check_line(d, n_gpus):
    assert d["impl"] == "reference" and d["n_gpus"] == n_gpus
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["higher_is_better"] is True
    assert d["vs_baseline"] is None and d["data"] == "synthetic" and d["scaling"] == "weak"
    assert d["config"]["workload"] == "tiny"
    c = d["cpu_baseline"]
    assert c["kind"] == "oracle" and c["value"] == d["value"] and c["cores"] >= 1 and c["sample"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_reference_arm_single_process():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "tiny",
                        "--steps", "2", "--warmup", "1", "--cpu-seconds", "1"], cwd=ROOT,
                       env=env(), capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = json_lines(r.stdout)
    assert len(lines) == 1
    check_line(lines[0], 1)


def test_reference_arm_two_ranks():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    r = subprocess.run([sys.executable, "-m", "torch.distributed.run", "--nnodes=1",
                        "--nproc-per-node", "2", "--master-addr", "127.0.0.1", "--master-port",
                        str(port), "bench.py", "--impl", "reference", "--gpus", "2",
                        "--workload", "tiny", "--steps", "1", "--warmup", "1",
                        "--cpu-seconds", "1"], cwd=ROOT, env=env(), capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = json_lines(r.stdout)
    assert len(lines) == 1
    check_line(lines[0], 2)


def test_cpu_baseline_parity_figure():
    """The CPU-baseline leg checks the bench's own log-probs on the tokens it
    samples: values equal to the oracle's are within tolerance, and a planted
    error of 0.05 in one context is reported."""
    import numpy as np
    import sys
    sys.path.insert(0, ROOT)
    import bench
    import hdl_synth
    import oracle
    wl = hdl_synth.generate(hdl_synth.SPECS["tiny"], device="cpu")
    W = oracle.widen(wl.w.numpy(), "f32")
    y = wl.targets.numpy()
    lp0 = oracle.target_logprobs(oracle.widen(wl.h_orig.numpy(), "f32"), W, y)
    lp1 = oracle.target_logprobs(oracle.widen(wl.h_hind.numpy(), "f32"), W, y)
    good = bench.cpu_oracle_sample(wl, 0.2, gpu_logp=(lp0, lp1))
    assert good["parity"]["within"] and good["parity"]["max_abs_err_logp"] < 1e-9
    assert good["parity"]["tokens"] > 0
    bad = bench.cpu_oracle_sample(wl, 0.2, gpu_logp=(lp0, lp1 + 0.05))
    assert not bad["parity"]["within"]
    assert abs(bad["parity"]["max_abs_err_logp"] - 0.05) < 1e-9
    assert "parity" not in bench.cpu_oracle_sample(wl, 0.1)
