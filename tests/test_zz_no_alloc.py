"""The allocation-free re-scoring entry point, called through the C ABI.

Some callers cannot allocate device memory while they run: plugin enqueue
callbacks of inference runtimes forbid it, processes whose device memory is
owned by a pooling allocator risk failure or fragmentation, and
latency-critical loops cannot afford the device synchronisation that
cudaMalloc/cudaFree may cause.  hdl_rescore_noalloc serves them from one
static 64 MiB device array.  These tests check that two calls in a row, on
different inputs, give what hdl_rescore gives on the same inputs (within the
log-probability tolerance of the parity tests), and that problems needing
more scratch than the array holds are refused before anything runs.

This file is collected last, so that a run stopping at its first failure has
already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

import hdl_synth
from tests.helpers import LP_ATOL, LP_RTOL


@pytest.fixture(scope="module")
def hdl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as m
    return m


def _noalloc(L, wl, lp0, lp1, delta, stream):
    scratch = ctypes.c_void_p(0)
    code = L.hdl_rescore_noalloc(
        ctypes.c_void_p(wl.h_orig.data_ptr()), ctypes.c_void_p(wl.h_hind.data_ptr()),
        ctypes.c_void_p(wl.w.data_ptr()), 0 if wl.spec.dtype == "bf16" else 1,
        ctypes.c_void_p(wl.targets.data_ptr()), wl.n_tokens, wl.spec.d, wl.spec.vocab,
        ctypes.c_void_p(lp0.data_ptr()), ctypes.c_void_p(lp1.data_ptr()),
        ctypes.c_void_p(delta.data_ptr()), ctypes.byref(scratch), ctypes.c_void_p(stream))
    return code, scratch.value


def _close(a, b):
    a = a.double().cpu().numpy()
    b = b.double().cpu().numpy()
    return bool(np.all(np.abs(a - b) <= LP_ATOL + LP_RTOL * np.abs(b)))


@pytest.mark.gpu
def test_noalloc_matches_rescore_on_two_calls(hdl):
    L = hdl.lib()
    stream = torch.cuda.current_stream().cuda_stream
    specs = [hdl_synth.small_spec("na1", n_roots=4, t_lo=300, t_hi=900, d=256, vocab=5000,
                                  seed=21),
             hdl_synth.small_spec("na2", n_roots=2, t_lo=100, t_hi=500, d=512, vocab=9000,
                                  seed=22)]
    first_scratch = None
    for spec in specs:                      # two calls in a row, different inputs
        wl = hdl_synth.generate(spec, device="cuda")
        r0, r1, rd, _ = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets)
        lp0 = torch.full_like(r0, float("nan"))
        lp1 = torch.full_like(r0, float("nan"))
        dl = torch.full_like(r0, float("nan"))
        code, scratch = _noalloc(L, wl, lp0, lp1, dl, stream)
        assert code == hdl.HDL_OK, hdl.hdl_status_string(code)
        assert scratch and scratch % 256 == 0
        if first_scratch is None:
            first_scratch = scratch
        assert scratch == first_scratch     # the one static array, every call
        raw = ctypes.c_uint32(0xFFFFFFFF)
        st = L.hdl_device_status(ctypes.c_void_p(scratch), hdl.HDL_STATIC_SCRATCH_BYTES,
                                 ctypes.c_void_p(stream), ctypes.byref(raw))
        assert st == hdl.HDL_OK and raw.value == 0
        assert _close(lp0, r0) and _close(lp1, r1)
        assert torch.all(torch.abs(dl - rd) <= 2 * LP_ATOL + LP_RTOL * (r0.abs() + r1.abs()))


def test_noalloc_refuses_oversized_problems(hdl):
    """Refused on the host, before any CUDA call (runs without a GPU)."""
    L = hdl.lib()
    P = ctypes.c_void_p(0x10000)
    n = 100_000   # at d = 4096, V = 152064 this needs ~228 MiB of scratch
    assert hdl.hdl_rescore_workspace_bytes(n, 4096, 152064) > hdl.HDL_STATIC_SCRATCH_BYTES
    code = L.hdl_rescore_noalloc(P, P, P, 0, P, n, 4096, 152064, P, P, None, None, None)
    assert code == hdl.HDL_ERR_UNSUPPORTED
    # shape errors are reported as by hdl_rescore
    assert L.hdl_rescore_noalloc(P, P, P, 0, P, 10, 100, 1000, P, P, None, None, None) == 2
    assert L.hdl_rescore_noalloc(P, P, P, 0, P, 0, 64, 1000, P, P, None, None, None) == 0
