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


def test_binding_rejects_short_and_mismatched_buffers(hdl):
    """The C entry points take every length from their scalar arguments, so
    the binding must refuse tensors shorter than those lengths, of another
    shape or on another device before it passes a pointer."""
    dev = "cuda"
    N, d, V = 64, 128, 512
    h = torch.zeros(N, d, dtype=torch.bfloat16, device=dev)
    w = torch.zeros(V, d, dtype=torch.bfloat16, device=dev)
    y = torch.zeros(N, dtype=torch.int32, device=dev)
    f = lambda n: torch.zeros(n, dtype=torch.float32, device=dev)
    bad_rescore = [
        dict(h_hind=h[:N - 1]),                                     # short second context
        dict(targets=y[:N - 1]),                                    # short targets
        dict(w_lmhead=torch.zeros(V, d + 64, dtype=torch.bfloat16, device=dev)),
        dict(h_hind=h.float()),                                     # mixed dtypes
        dict(logp_orig=f(N - 1)),                                   # short output
        dict(delta=f(N - 1)),
        dict(targets=y.cpu()),                                      # host tensor
    ]
    for kw in bad_rescore:
        args = dict(h_orig=h, h_hind=h, w_lmhead=w, targets=y)
        args.update(kw)
        with pytest.raises((ValueError, TypeError)):
            hdl.hdl_rescore(**args)
        with pytest.raises((ValueError, TypeError)):
            hdl.hdl_rescore_ex(**args)
    with pytest.raises(ValueError):
        hdl.hdl_rescore_noalloc(h, h[:N - 1], w, y, f(N), f(N))
    with pytest.raises(ValueError):
        hdl.hdl_rescore_shard(h, h, w, y[:N - 1], 0)
    with pytest.raises(ValueError):
        hdl.hdl_rescore_shard(h, h, w, y, 0, stats=f(2 * N * 4 - 1))
    offs = torch.tensor([0, 30, 64], dtype=torch.int64, device=dev)
    u8 = lambda n: torch.ones(n, dtype=torch.uint8, device=dev)
    i32 = lambda *s: torch.zeros(*s, dtype=torch.int32, device=dev)
    for kw in (dict(valid=u8(N - 1)), dict(branch_pos=i32(2, 3)), dict(n_selected=i32(1)),
               dict(branch_delta=f(7))):
        args = dict(delta=f(N), valid=None, root_offsets=offs, k=4)
        args.update(kw)
        with pytest.raises(ValueError):
            hdl.hdl_select_branches(**args)
    with pytest.raises(ValueError):
        hdl.hdl_assign_continuations(i32(1), i32(2, 4), i32(2), n_cont=8)
    with pytest.raises(ValueError):
        hdl.hdl_assign_continuations(i32(2), i32(2, 4), i32(3), n_cont=8)
    coffs = torch.tensor([0, 10, 20], dtype=torch.int64, device=dev)
    with pytest.raises(ValueError):
        hdl.hdl_suffix_mask(i32(3), coffs, u8(20))                  # offsets one short
    with pytest.raises(ValueError):
        hdl.hdl_suffix_mask(i32(2), coffs, u8(19), mask=u8(20))     # valid shorter than mask
    toffs = torch.tensor([0, 30, 64], dtype=torch.int64, device=dev)
    goffs = torch.tensor([0, 2], dtype=torch.int32, device=dev)
    good = dict(logp_new=f(N), logp_old=f(N), mask=u8(N), traj_offsets=toffs, rewards=f(2),
                group_offsets=goffs)
    for kw in (dict(logp_old=f(N - 1)), dict(mask=u8(N - 1)), dict(rewards=f(1)),
               dict(advantages=f(1)), dict(grad=f(N - 1)), dict(stats=f(3))):
        args = dict(good)
        args.update(kw)
        with pytest.raises(ValueError):
            hdl.hdl_grpo_loss(**args)
    torch.cuda.synchronize()
    adv, grad, st = hdl.hdl_grpo_loss(**good)                       # the well-formed call runs
    assert int(st[1].item()) == N
