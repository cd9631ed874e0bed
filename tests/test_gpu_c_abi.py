"""libhdl used from plain C: tests/c/abi_from_c.c is compiled with gcc
against include/hdl.h, linked to libhdl.so and the CUDA runtime, and run on
a small problem; its log-probs and branch points must equal the Python
binding's bit for bit, and its argument-error checks must pass."""
import os
import shutil
import subprocess

import numpy as np
import pytest
import torch

import hdl_synth

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def hdl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as m
    return m


def test_c_program_matches_binding(hdl, tmp_path):
    cuda = "/usr/local/cuda"
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    exe = str(tmp_path / "abi_from_c")
    libdir = os.path.dirname(hdl.library_path())
    subprocess.run([cc, "-O2", "-o", exe, os.path.join(ROOT, "tests", "c", "abi_from_c.c"),
                    "-I" + os.path.join(ROOT, "include"), "-I" + cuda + "/include",
                    "-L" + libdir, "-lhdl", "-L" + cuda + "/lib64", "-lcudart",
                    "-Wl,-rpath," + libdir + ":" + cuda + "/lib64"], check=True)
    spec = hdl_synth.small_spec("c", n_roots=3, t_lo=100, t_hi=400, d=256, vocab=5000, k=4,
                                seed=31)
    wl = hdl_synth.generate(spec, device="cuda")
    N, R, k = wl.n_tokens, spec.n_roots, spec.k
    inp = tmp_path / "in.bin"
    with open(inp, "wb") as f:
        for t in (wl.h_orig, wl.h_hind, wl.w):
            f.write(t.cpu().view(torch.int16).numpy().tobytes())
        f.write(wl.targets.cpu().numpy().tobytes())
        f.write(wl.root_offsets.cpu().numpy().tobytes())
    out = tmp_path / "out.bin"
    r = subprocess.run([exe, str(inp), str(out), str(N), str(spec.d), str(spec.vocab), str(R),
                        str(k)], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, (r.returncode, r.stdout, r.stderr)
    raw = np.fromfile(out, dtype=np.float32, count=2 * N)
    bp_c = np.fromfile(out, dtype=np.int32, offset=8 * N).reshape(R, k)
    lp0, lp1, de, _ = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets)
    bp, ns, bd = hdl.hdl_select_branches(de, None, wl.root_offsets, k)
    assert np.array_equal(raw[:N], lp0.cpu().numpy())
    assert np.array_equal(raw[N:], lp1.cpu().numpy())
    assert np.array_equal(bp_c, bp.cpu().numpy())
