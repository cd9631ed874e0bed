"""The C ABI without a GPU: libhdl.so loads, exports every symbol that
include/hdl.h declares, and rejects bad arguments on the host before it
touches CUDA (each case here returns before the first CUDA call)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "hdl.h")


@pytest.fixture(scope="module")
def L():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as hdl
    return hdl.lib()


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"HDL_API\s+[\w\s\*]*?\b(hdl_\w+)\s*\(", text)))


def test_header_declares_the_entry_points():
    syms = declared_symbols()
    for name in ("hdl_rescore", "hdl_select_branches", "hdl_assign_continuations",
                 "hdl_suffix_mask", "hdl_rescore_workspace_bytes", "hdl_device_status"):
        assert name in syms


def test_library_exports_every_declared_symbol(L):
    for name in declared_symbols():
        assert hasattr(L, name), name


def test_only_declared_symbols_exported(L):
    import subprocess
    out = subprocess.run(["nm", "-D", "--defined-only", L._name], capture_output=True,
                         text=True).stdout
    exported = sorted({l.split()[-1] for l in out.splitlines()
                       if " T " in l and l.split()[-1].startswith("hdl_")})
    assert exported == declared_symbols()


def test_abi_version_and_names(L):
    import paper_2609_36864_gb300 as hdl
    assert hdl.hdl_abi_version() == 2
    assert hdl.hdl_status_string(0) == "HDL_OK"
    assert hdl.hdl_status_string(5) == "HDL_ERR_TIMEOUT"
    assert hdl.hdl_status_string(99) == "HDL_ERR_UNKNOWN"


def _chunk_tiles(n, d, V, esize):
    """Vocabulary tiles per chunk: from 16, halved while the H tiles of a group
    of 32 M-tiles plus the W tiles of the 76 / 16 chunks in flight exceed
    70 MB, then while there are fewer than 1216 work units."""
    cdiv = lambda a, b: -(-a // b)
    num_m, nvt, tpc = 2 * cdiv(n, 128), cdiv(V, 256), 16
    row = d * esize
    while tpc > 1 and 32 * 128 * row + (2 * 76 / 32) * tpc * 256 * row > 70e6:
        tpc //= 2
    while tpc > 1 and num_m * cdiv(nvt, tpc) < 1216:
        tpc //= 2
    return tpc


def _ws_formula(n, d, V, esize=2):
    """status (256 B) + merge counters (4 per 128-token tile) + target logits
    + per-(chunk, row) partials."""
    cdiv = lambda a, b: -(-a // b)
    chunks = cdiv(cdiv(V, 256), _chunk_tiles(n, d, V, esize))
    done = cdiv(cdiv(n, 128) * 4 * 4, 256) * 256
    zt = cdiv(2 * n * 4, 256) * 256
    return 256 + done + zt + chunks * 2 * n * 8


@pytest.mark.parametrize("n,d,V", [(0, 64, 1), (1, 64, 1), (2048, 256, 4096),
                                   (18000, 2048, 32000), (327680, 5120, 152064),
                                   (5, 128, 4097), (8192, 4096, 32000), (1000, 64, 152064)])
def test_workspace_bytes(L, n, d, V):
    import paper_2609_36864_gb300 as hdl
    assert hdl.hdl_rescore_workspace_bytes(n, d, V, hdl.HDL_BF16) == _ws_formula(n, d, V, 2)
    assert hdl.hdl_rescore_workspace_bytes(n, d, V, hdl.HDL_F32) == _ws_formula(n, d, V, 4)


def test_workspace_bytes_rejects_bad_shapes(L):
    import paper_2609_36864_gb300 as hdl
    assert hdl.hdl_rescore_workspace_bytes(10, 100, 1000, 0) == 0      # d % 64
    assert hdl.hdl_rescore_workspace_bytes(-1, 64, 1000, 0) == 0
    assert hdl.hdl_rescore_workspace_bytes(10, 64, 0, 0) == 0
    assert hdl.hdl_rescore_workspace_bytes(10, 64, 10, 7) == 0          # dtype


P = ctypes.c_void_p(0x10000)   # aligned stand-in pointers: never dereferenced


def _rescore(L, n=16, d=64, V=100, dt=0, ws=P, wsb=1 << 40, h=P, t=P, lp=P):
    return L.hdl_rescore(h, P, P, dt, t, n, d, V, lp, P, None, ws, wsb, None)


def test_rescore_argument_errors(L):
    assert _rescore(L, d=100) == 2          # d % 64 != 0 -> UNSUPPORTED
    assert _rescore(L, d=65536 + 64) == 2
    assert _rescore(L, n=-1) == 1
    assert _rescore(L, V=0) == 1
    assert _rescore(L, dt=3) == 1
    assert _rescore(L, h=None) == 1
    assert _rescore(L, t=None) == 1
    assert _rescore(L, lp=None) == 1
    assert _rescore(L, h=ctypes.c_void_p(0x10008)) == 1     # TMA needs 16-B alignment
    assert _rescore(L, ws=None) == 3
    assert _rescore(L, ws=ctypes.c_void_p(0x10010)) == 3    # workspace 256-B aligned
    assert _rescore(L, wsb=100) == 3
    assert _rescore(L, n=0) == 0            # empty: no launch


def _select(L, n_roots=2, k=4, opts=(0, 0, 0, 0), offs=P, delta=P):
    import paper_2609_36864_gb300 as hdl
    o = hdl._SelectOpts(*opts)
    return L.hdl_select_branches(delta, None, 100, offs, n_roots, k, ctypes.byref(o), P, P,
                                 None, None)


def test_select_argument_errors(L):
    assert _select(L, k=17) == 2
    assert _select(L, k=-1) == 1
    assert _select(L, n_roots=-1) == 1
    assert _select(L, opts=(-1, 0, 0, 0)) == 1
    assert _select(L, opts=(2, 2, 0, 0)) == 1
    assert _select(L, offs=None) == 1
    assert _select(L, offs=ctypes.c_void_p(0x10004)) == 1
    assert _select(L, delta=None) == 1
    assert _select(L, n_roots=0) == 0


def test_assign_argument_errors(L):
    assert L.hdl_assign_continuations(P, P, 2, 17, P, 1, P, 10, None) == 2
    assert L.hdl_assign_continuations(P, P, -1, 4, P, 1, P, 10, None) == 1
    assert L.hdl_assign_continuations(None, P, 2, 4, P, 1, P, 10, None) == 1
    assert L.hdl_assign_continuations(P, P, 2, 4, P, 1, P, -1, None) == 1
    assert L.hdl_assign_continuations(P, P, 0, 4, P, 1, P, 10, None) == 0
    assert L.hdl_assign_continuations(P, P, 2, 4, P, 1, P, 0, None) == 0


def test_mask_argument_errors(L):
    assert L.hdl_suffix_mask(P, P, -1, None, P, 10, None) == 1
    assert L.hdl_suffix_mask(P, P, 3, None, P, -1, None) == 1
    assert L.hdl_suffix_mask(None, P, 3, None, P, 10, None) == 1
    assert L.hdl_suffix_mask(P, ctypes.c_void_p(0x10004), 3, None, P, 10, None) == 1
    assert L.hdl_suffix_mask(P, P, 0, None, P, 10, None) == 0
    assert L.hdl_suffix_mask(P, P, 3, None, P, 0, None) == 0


def test_device_status_argument_errors(L):
    assert L.hdl_device_status(None, 256, None, None) == 1
    assert L.hdl_device_status(P, 0, None, None) == 1


def test_product_path_fails_loudly_without_library(monkeypatch, tmp_path):
    import paper_2609_36864_gb300 as hdl
    monkeypatch.setattr(hdl, "_lib", None)
    monkeypatch.setattr(hdl, "library_path", lambda: str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="libhdl.so not found"):
        hdl.hdl_abi_version()


def test_rescore_ex_options_and_workspace(L):
    import paper_2609_36864_gb300 as hdl
    n, d, V = 5000, 256, 9000
    base = hdl.hdl_rescore_workspace_bytes(n, d, V)
    assert hdl.hdl_rescore_ex_workspace_bytes(n, d, V) == base
    ent = hdl.hdl_rescore_ex_workspace_bytes(n, d, V, entropy=True)
    cdiv = lambda a, b: -(-a // b)
    assert ent == cdiv(base, 256) * 256 + cdiv(cdiv(V, 256), _chunk_tiles(n, d, V, 2)) * 2 * n * 4
    o = hdl._RescoreOpts(None, None, 0, 2, 0)          # unknown fault bit
    assert L.hdl_rescore_ex(P, P, P, 0, P, 16, 64, 100, P, P, None, ctypes.byref(o), P,
                            1 << 40, None) == 1
    o = hdl._RescoreOpts(0x10002, None, 0, 0, 0)       # misaligned entropy output
    assert L.hdl_rescore_ex(P, P, P, 0, P, 16, 64, 100, P, P, None, ctypes.byref(o), P,
                            1 << 40, None) == 1
    o = hdl._RescoreOpts(0x10000, None, 0, 0, 0)       # entropy needs the larger workspace
    small = hdl.hdl_rescore_workspace_bytes(16, 64, 100)
    assert L.hdl_rescore_ex(P, P, P, 0, P, 16, 64, 100, P, P, None, ctypes.byref(o), P,
                            small, None) == 3


def test_binding_allocates_outputs_at_the_inputs_phase():
    """Outputs the binding allocates (GRPO gradient, suffix mask) start at the
    same address residue mod 16 as the input they stream with, so sliced
    inputs keep the kernels' 16-byte vector paths."""
    import torch
    from paper_2609_36864_gb300 import _empty_like_phase
    for dt in (torch.float32, torch.uint8):
        es = torch.empty(0, dtype=dt).element_size()
        for off in range(16 // es):
            like = torch.empty(100 + off, dtype=dt)[off:]
            out = _empty_like_phase(37, dt, like, 16)
            assert out.numel() == 37 and out.dtype == dt
            assert out.data_ptr() % 16 == like.data_ptr() % 16
