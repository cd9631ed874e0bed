"""The five workloads (tiny, math, code, agent, roofline sweep) at their full
sizes, in the launch configuration the bench times, and the math workload
with fp32 states (the tf32 path at a large shape).

tiny and math: the oracle scores every token, so log-probs, scores and the
end-to-end branch sets are compared in full.  code, agent and the sweep: the
oracle scores sampled tokens one by one (first, last, random), and selection,
allocation and masks are compared bit-exactly on the device's own scores; on
top of that it scores whole roots (code: the first and the last; agent: the
shortest, to bound the fp64 work; three sweep vocabularies: the last root),
and on those every token's log-probs and |Delta| and the root's branch set
(Section 3.2: the k highest-scoring valid positions) are compared with the
oracle's -- branch sets equal except at positions whose oracle score is
within 2e-3 of the root's k-th."""
import dataclasses

import numpy as np
import pytest
import torch

import hdl_synth
import oracle
from tests.helpers import (assert_logp_close, check_selection_band, oracle_logprobs,
                           sample_rows, to_f64)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hdl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as m
    return m


def run_path(hdl, wl):
    k = wl.spec.k
    lp0, lp1, delta, ws = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets)
    bp, ns, bd = hdl.hdl_select_branches(delta, wl.valid, wl.root_offsets, k)
    cb = hdl.hdl_assign_continuations(ns, bp, wl.conts_per_root,
                                      n_cont=wl.cont_offsets.numel() - 1)
    mask = hdl.hdl_suffix_mask(cb, wl.cont_offsets, wl.cont_valid)
    code, raw = hdl.hdl_device_status(ws)
    assert code == hdl.HDL_OK, (code, hex(raw))
    return dict(lp0=lp0.cpu().numpy(), lp1=lp1.cpu().numpy(), delta=delta.cpu().numpy(),
                bp=bp.cpu().numpy(), ns=ns.cpu().numpy(), bd=bd.cpu().numpy(),
                cb=cb.cpu().numpy(), mask=mask.cpu().numpy())


def check_downstream_exact(wl, out):
    """Selection / allocation / mask of the oracle on the device's scores."""
    valid = wl.valid.cpu().numpy()
    offs = wl.root_offsets.cpu().numpy()
    d = out["delta"].astype(np.float64)
    pos, nsel, val = oracle.select_branches(d, valid, offs, wl.spec.k)
    assert np.array_equal(out["ns"], nsel)
    assert np.array_equal(out["bp"], pos)
    assert np.array_equal(out["bd"].astype(np.float64), val, equal_nan=True)
    cb = oracle.assign_continuations(nsel, pos, wl.conts_per_root.cpu().numpy())
    assert np.array_equal(out["cb"], cb)
    m = oracle.suffix_mask(cb, wl.cont_offsets.cpu().numpy(), wl.cont_valid.cpu().numpy())
    assert np.array_equal(out["mask"], m)
    # invalid (observation) tokens are never branch points
    for r in range(len(offs) - 1):
        for t in out["bp"][r, :out["ns"][r]]:
            assert valid[offs[r] + t]


@pytest.mark.parametrize("name", ["tiny", "math"])
def test_workload_full_oracle(hdl, name):
    wl = hdl_synth.generate(hdl_synth.SPECS[name], device="cuda")
    out = run_path(hdl, wl)
    W = to_f64(wl.w)
    y = wl.targets.cpu().numpy()
    r0 = oracle_logprobs(to_f64(wl.h_orig), W, y)
    r1 = oracle_logprobs(to_f64(wl.h_hind), W, y)
    assert_logp_close(out["lp0"], r0, name + " orig")
    assert_logp_close(out["lp1"], r1, name + " hind")
    rd = oracle.hindsight_divergence(r1, r0)
    # |Delta| inherits both contexts' errors
    err = np.abs(out["delta"] - rd)
    assert np.all(err <= 2e-3 + 1e-3 * (np.abs(r0) + np.abs(r1))), err.max()
    check_selection_band(out["bp"], out["ns"], rd, wl.valid.cpu().numpy(),
                         wl.root_offsets.cpu().numpy(), wl.spec.k)
    check_downstream_exact(wl, out)


# the last entry is four times the largest workload: 2^20 tokens per context,
# 4.3 G elements (8.6 GB) per context, past every 32-bit element count
SAMPLED = ["code", "agent", "math_f32", ("sweep", 32000, 8192), ("sweep", 256000, 262144),
           ("sweep", 128256, 131072), ("sweep", 32000, 1 << 20)]


def sampled_spec(which):
    if isinstance(which, tuple):
        return hdl_synth.sweep_spec(which[1], which[2])
    if which.endswith("_f32"):   # fp32 hidden states and LM head: tf32 products
        return dataclasses.replace(hdl_synth.SPECS[which[:-4]], name=which, dtype="f32")
    return hdl_synth.SPECS[which]


# whole roots scored by the oracle, per workload: "first_last", "shortest", "last"
WHOLE_ROOTS = {"code": "first_last", "agent": "shortest", ("sweep", 32000, 1 << 20): "last",
               ("sweep", 128256, 131072): "last", ("sweep", 256000, 262144): "last"}


def whole_roots(wl, how):
    R = wl.spec.n_roots
    if how == "first_last":
        return [0, R - 1]
    if how == "shortest":
        return [int(np.argmin(wl.lengths))]
    return [R - 1]


def check_whole_roots(wl, out, roots, W):
    """Every token of each root in ``roots``, both contexts, against the
    oracle, and the root's branch set against the oracle's on the oracle's
    scores (the end-to-end band check)."""
    offs = wl.root_offsets.cpu().numpy()
    valid = wl.valid.cpu().numpy()
    y_all = wl.targets.cpu().numpy()
    k = wl.spec.k
    for r in roots:
        a, b = int(offs[r]), int(offs[r + 1])
        r0 = oracle_logprobs(to_f64(wl.h_orig[a:b]), W, y_all[a:b], block=256)
        r1 = oracle_logprobs(to_f64(wl.h_hind[a:b]), W, y_all[a:b], block=256)
        what = f"{wl.spec.name} root {r} ({b - a} tokens)"
        assert_logp_close(out["lp0"][a:b], r0, what + " orig")
        assert_logp_close(out["lp1"][a:b], r1, what + " hind")
        rd = oracle.hindsight_divergence(r1, r0)
        err = np.abs(out["delta"][a:b] - rd)
        assert np.all(err <= 2e-3 + 1e-3 * (np.abs(r0) + np.abs(r1))), (what, err.max())
        check_selection_band(out["bp"][r:r + 1], out["ns"][r:r + 1], rd, valid[a:b],
                             np.array([0, b - a]), k)


@pytest.mark.parametrize("which", SAMPLED, ids=lambda w: w if isinstance(w, str) else
                         f"sweep_V{w[1]}_N{w[2]}")
def test_workload_sampled(hdl, which):
    spec = sampled_spec(which)
    wl = hdl_synth.generate(spec, device="cuda")
    out = run_path(hdl, wl)
    rows = sample_rows(wl.n_tokens, 40, seed=spec.d)
    idx = torch.from_numpy(rows).cuda()
    W = to_f64(wl.w)
    y = wl.targets.cpu().numpy()[rows]
    r0 = oracle.target_logprobs(to_f64(wl.h_orig.index_select(0, idx)), W, y)
    r1 = oracle.target_logprobs(to_f64(wl.h_hind.index_select(0, idx)), W, y)
    assert_logp_close(out["lp0"][rows], r0, spec.name + " orig")
    assert_logp_close(out["lp1"][rows], r1, spec.name + " hind")
    if which in WHOLE_ROOTS:
        check_whole_roots(wl, out, whole_roots(wl, WHOLE_ROOTS[which]), W)
    del W
    check_downstream_exact(wl, out)
    # properties that hold at any size
    assert np.all(out["lp0"] <= 1e-5) and np.all(out["lp1"] <= 1e-5)
    assert np.all(np.isfinite(out["delta"])) and np.all(out["delta"] >= 0)


@pytest.mark.parametrize("name", ["tiny", "math"])
def test_workload_entropy_selector(hdl, name):
    """The Entropy selector of Section 4.1: rank positions by the entropy of
    the next-token distribution under the original context, through the same
    selection kernel; branch sets match the oracle's within the band."""
    wl = hdl_synth.generate(hdl_synth.SPECS[name], device="cuda")
    lp0, lp1, de, e0, _, ws = hdl.hdl_rescore_ex(wl.h_orig, wl.h_hind, wl.w, wl.targets)
    bp, ns, bd = hdl.hdl_select_branches(e0, wl.valid, wl.root_offsets, wl.spec.k)
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
    ref = oracle.next_token_entropy(to_f64(wl.h_orig), to_f64(wl.w)) if name == "tiny" else \
        np.concatenate([oracle.next_token_entropy(to_f64(wl.h_orig[s:s + 2048]), to_f64(wl.w))
                        for s in range(0, wl.n_tokens, 2048)])
    assert_logp_close(e0.cpu().numpy(), ref, name + " entropy")
    check_selection_band(bp.cpu().numpy(), ns.cpu().numpy(), ref, wl.valid.cpu().numpy(),
                         wl.root_offsets.cpu().numpy(), wl.spec.k)


def test_random_small_workloads_end_to_end(hdl):
    """12 seeded random small workloads through the whole path (re-scoring,
    selection, allocation, masks): every token's log-probs and |Delta|
    against the oracle, branch sets within the band of the root's k-th
    oracle score (Section 3.2), and selection / allocation / masks bit-exact
    on the device's scores."""
    rng = np.random.default_rng(4242)
    for case in range(12):
        T_lo = int(rng.integers(1, 400))
        spec = hdl_synth.small_spec(
            f"e2e{case}", n_roots=int(rng.integers(1, 13)), t_lo=T_lo,
            t_hi=T_lo + int(rng.integers(0, 1200)), d=64 * int(rng.integers(1, 9)),
            vocab=int(rng.integers(50, 20001)), dtype="f32" if case % 5 == 4 else "bf16",
            k=int(rng.integers(1, 17)), pert_frac=float(rng.choice([0.01, 0.05, 0.2])),
            pert_mode=str(rng.choice(["uniform", "spans", "valid"])),
            invalid_frac=float(rng.choice([0.0, 0.2])),
            conts_per_root=int(rng.integers(1, 9)), seed=500 + case)
        wl = hdl_synth.generate(spec, device="cuda")
        out = run_path(hdl, wl)
        W = to_f64(wl.w)
        y = wl.targets.cpu().numpy()
        r0 = oracle_logprobs(to_f64(wl.h_orig), W, y)
        r1 = oracle_logprobs(to_f64(wl.h_hind), W, y)
        assert_logp_close(out["lp0"], r0, f"{spec.name} orig")
        assert_logp_close(out["lp1"], r1, f"{spec.name} hind")
        rd = oracle.hindsight_divergence(r1, r0)
        assert np.all(np.abs(out["delta"] - rd) <= 2e-3 + 1e-3 * (np.abs(r0) + np.abs(r1)))
        check_selection_band(out["bp"], out["ns"], rd, wl.valid.cpu().numpy(),
                             wl.root_offsets.cpu().numpy(), spec.k)
        check_downstream_exact(wl, out)
