"""Vocabulary-parallel re-scoring (a tensor-parallel LM head) emulated on one
GPU: W is cut into uneven shards, each shard's statistics come from
hdl_rescore_shard, and hdl_merge_vocab_shards must give the log-probs, |Delta|
and entropies of the unsharded call and of the oracle."""
import numpy as np
import pytest
import torch

import hdl_synth
import oracle
from tests.helpers import assert_logp_close, oracle_logprobs, to_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hdl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as m
    return m


@pytest.mark.parametrize("n,d,V,cuts,dt", [
    (700, 256, 9000, [2500, 2501], "bf16"),      # a one-column shard in the middle
    (300, 128, 4096, [2048], "bf16"),
    (129, 64, 1000, [1, 500, 999], "bf16"),
    (200, 256, 5000, [1700, 3400], "f32"),
])
def test_vocab_shards_merge_to_unsharded(hdl, n, d, V, cuts, dt):
    spec = hdl_synth.small_spec("shard", n_roots=1, t_lo=n, t_hi=n, d=d, vocab=V, dtype=dt,
                                seed=n + len(cuts))
    wl = hdl_synth.generate(spec, device="cuda")
    bounds = [0] + cuts + [V]
    stats = torch.empty((len(bounds) - 1, 2, n, 4), dtype=torch.float32, device="cuda")
    for p in range(len(bounds) - 1):
        lo, hi = bounds[p], bounds[p + 1]
        hdl.hdl_rescore_shard(wl.h_orig, wl.h_hind, wl.w[lo:hi].contiguous(), wl.targets, lo,
                              stats=stats[p])
    lp0, lp1, de, e0, e1 = hdl.hdl_merge_vocab_shards(stats)
    # exactly one shard owns each target
    owned = (~torch.isnan(stats[:, 0, :, 2])).sum(0)
    assert torch.all(owned == 1)
    full = hdl.hdl_rescore_ex(wl.h_orig, wl.h_hind, wl.w, wl.targets, want_entropy_hind=True)
    for a, b in zip((lp0, lp1, e0, e1), (full[0], full[1], full[3], full[4])):
        assert_logp_close(a.cpu().numpy(), b.double().cpu().numpy(), "shards vs full")
    W = to_f64(wl.w)
    y = wl.targets.cpu().numpy()
    r0 = oracle_logprobs(to_f64(wl.h_orig), W, y)
    r1 = oracle_logprobs(to_f64(wl.h_hind), W, y)
    assert_logp_close(lp0.cpu().numpy(), r0, "shards orig")
    assert_logp_close(lp1.cpu().numpy(), r1, "shards hind")
    assert_logp_close(e0.cpu().numpy(), oracle.next_token_entropy(to_f64(wl.h_orig), W), "H")
    assert torch.equal(de, (lp1 - lp0).abs())


def test_vocab_shards_missing_target_is_nan(hdl):
    spec = hdl_synth.small_spec("shard2", n_roots=1, t_lo=200, t_hi=200, d=64, vocab=1000,
                                seed=3)
    wl = hdl_synth.generate(spec, device="cuda")
    stats, _ = hdl.hdl_rescore_shard(wl.h_orig, wl.h_hind, wl.w[:600].contiguous(),
                                     wl.targets, 0)
    lp0, lp1, de, e0, e1 = hdl.hdl_merge_vocab_shards(stats[None])
    y = wl.targets.cpu()
    assert torch.equal(torch.isnan(lp0).cpu(), y >= 600)
    assert torch.all(torch.isfinite(e0))      # the shard's own entropy is still defined
