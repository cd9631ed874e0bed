"""Failure detection on the GPU without faulting it: every pipeline wait in
the re-scoring kernel is bounded.  The test hook makes the copy producer issue
nothing (a barrier that nothing will complete), so a wait runs out after a
short limit, the kernel records HDL_ERR_TIMEOUT in the workspace status word
and returns; the context stays usable and the next call is exact."""
import numpy as np
import pytest
import torch

import hdl_synth
from tests.helpers import assert_logp_close, oracle_logprobs, to_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hdl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as m
    return m


@pytest.mark.parametrize("entropy", [False, True])
def test_stalled_pipeline_reports_timeout_and_context_survives(hdl, entropy):
    spec = hdl_synth.small_spec("stall", n_roots=2, t_lo=200, t_hi=300, d=256, vocab=3000,
                                seed=5)
    wl = hdl_synth.generate(spec, device="cuda")
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    out = hdl.hdl_rescore_ex(wl.h_orig, wl.h_hind, wl.w, wl.targets, want_entropy=entropy,
                             wait_timeout_ns=50_000_000, fault_inject=1)
    t1.record()
    code, raw = hdl.hdl_device_status(out[-1])
    assert code == hdl.HDL_ERR_TIMEOUT, (code, hex(raw))
    assert raw & 1 and ((raw >> 8) & 0xFF) in (2, 3)     # MMA issuer or epilogue gave up
    assert t0.elapsed_time(t1) < 5000                     # bounded by the 50 ms limit
    # the context is intact: the same call without the hook is exact
    lp0, lp1, delta, ws = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets,
                                          workspace=out[-1])
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
    W = to_f64(wl.w)
    y = wl.targets.cpu().numpy()
    assert_logp_close(lp0.cpu().numpy(), oracle_logprobs(to_f64(wl.h_orig), W, y), "after")
    assert_logp_close(lp1.cpu().numpy(), oracle_logprobs(to_f64(wl.h_hind), W, y), "after")
