"""Re-scoring parity (Section 3.1-3.2): the tcgen05 kernel against the fp64
oracle, element by element, on shapes that cover every tile edge."""
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


def run_and_check(hdl, wl, what):
    lp0, lp1, delta, ws = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets)
    code, raw = hdl.hdl_device_status(ws)
    assert code == hdl.HDL_OK, (code, hex(raw))
    W = to_f64(wl.w)
    y = wl.targets.cpu().numpy()
    r0 = oracle_logprobs(to_f64(wl.h_orig), W, y)
    r1 = oracle_logprobs(to_f64(wl.h_hind), W, y)
    e0 = assert_logp_close(lp0.cpu().numpy(), r0, what + " orig")
    e1 = assert_logp_close(lp1.cpu().numpy(), r1, what + " hind")
    d = delta.cpu().numpy().astype(np.float64)
    assert np.array_equal(d, np.abs(lp1.cpu().numpy() - lp0.cpu().numpy()).astype(np.float64))
    # and against the oracle's |Delta| (Eq. div), which inherits both contexts' errors
    rd = np.abs(r1 - r0)
    assert np.all(np.abs(d - rd) <= 2e-3 + 1e-3 * (np.abs(r0) + np.abs(r1))), \
        (what, np.abs(d - rd).max())
    return max(e0, e1), r0, r1, d


# (tokens, d, V, dtype): rows around the 128-row tile, vocabularies around the
# 256-column tile and the 4096-column chunk, several K steps.
SHAPES = [
    (1, 64, 1, "bf16"),        # one row, one word: log p = 0
    (5, 64, 300, "bf16"),      # one partial vocabulary tile
    (127, 128, 256, "bf16"),
    (128, 128, 512, "bf16"),
    (129, 192, 257, "bf16"),   # ragged rows and a 1-column last tile
    (300, 256, 4097, "bf16"),  # second chunk holds a single column
    (700, 512, 9000, "bf16"),
    (1000, 1024, 8192, "bf16"),
    (200, 256, 5000, "f32"),   # tf32 path
    (513, 64, 4096, "f32"),
    (3, 256, 152064, "bf16"),  # decode-like: a few tokens, a full vocabulary (one tile per unit)
]


@pytest.mark.parametrize("n,d,V,dt", SHAPES)
def test_rescore_shapes(hdl, n, d, V, dt):
    spec = hdl_synth.small_spec(f"s{n}_{d}_{V}", n_roots=1, t_lo=n, t_hi=n, d=d, vocab=V,
                                dtype=dt, seed=n + V)
    wl = hdl_synth.generate(spec, device="cuda")
    err, r0, _, _ = run_and_check(hdl, wl, str((n, d, V, dt)))
    if V == 1:
        assert np.all(r0 == 0.0)


@pytest.mark.parametrize("V", [257, 1000, 4097, 32000])
def test_rescore_targets_at_the_vocabulary_edges(hdl, V):
    """Targets in the first column, the last column (inside the masked tail
    of a partial 256-column tile), the last column of a full tile and the
    first of the next, and the first and last columns of a vocabulary chunk:
    every gather position the epilogue special-cases."""
    spec = hdl_synth.small_spec(f"edge{V}", n_roots=1, t_lo=260, t_hi=260, d=128, vocab=V,
                                seed=V)
    wl = hdl_synth.generate(spec, device="cuda")
    cols = [0, V - 1, min(255, V - 1), min(256, V - 1), min(4095, V - 1), min(4096, V - 1),
            V // 2]
    y = torch.tensor([cols[i % len(cols)] for i in range(wl.n_tokens)], dtype=torch.int32,
                     device="cuda")
    wl.targets.copy_(y)
    run_and_check(hdl, wl, f"edges V={V}")


def test_rescore_identical_contexts_bitwise(hdl):
    """Delta = 0 exactly when both contexts carry the same hidden states, and
    the two log-prob rows are bit-identical (same arithmetic for both)."""
    spec = hdl_synth.small_spec("same", n_roots=2, t_lo=300, t_hi=400, d=256, vocab=6000)
    wl = hdl_synth.generate(spec, device="cuda")
    lp0, lp1, delta, ws = hdl.hdl_rescore(wl.h_orig, wl.h_orig.clone(), wl.w, wl.targets)
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
    assert torch.equal(lp0, lp1)
    assert torch.all(delta == 0)


def test_rescore_invariants(hdl):
    """log p <= 0 and the normaliser is shared: summing p over every target
    of one row gives 1."""
    V, d = 3000, 128
    g = torch.Generator(device="cuda").manual_seed(3)
    w = (torch.randn(V, d, generator=g, device="cuda") * 0.05).to(torch.bfloat16)
    h = torch.randn(1, d, generator=g, device="cuda").to(torch.bfloat16).repeat(V, 1)
    y = torch.arange(V, dtype=torch.int32, device="cuda")
    lp0, lp1, _, _ = hdl.hdl_rescore(h, h, w, y)
    lp = lp0.double()
    assert torch.all(lp <= 1e-6)
    assert abs(torch.exp(lp).sum().item() - 1.0) < 1e-4


def test_rescore_bad_target_reported(hdl):
    spec = hdl_synth.small_spec("bad", n_roots=1, t_lo=50, t_hi=50, d=64, vocab=500)
    wl = hdl_synth.generate(spec, device="cuda")
    y = wl.targets.clone()
    y[7] = 500
    y[9] = -1
    lp0, lp1, delta, ws = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, y)
    code, raw = hdl.hdl_device_status(ws)
    assert code == hdl.HDL_ERR_BAD_TARGET and (raw & 2)
    bad = torch.isnan(lp0).cpu()
    assert bad[7] and bad[9] and bad.sum() == 2
    # the next call on the same workspace starts from a clear status word
    lp0, lp1, delta, ws = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets, workspace=ws)
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK


def test_rescore_outputs_independent_of_stream_and_repeat(hdl):
    spec = hdl_synth.small_spec("rep", n_roots=3, t_lo=100, t_hi=400, d=256, vocab=5000)
    wl = hdl_synth.generate(spec, device="cuda")
    a = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        b = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets, stream=s)
    s.synchronize()
    for x, y in zip(a[:3], b[:3]):
        assert torch.equal(x, y)


_MODE_SCRIPT = r"""
import sys, numpy as np, torch
sys.path.insert(0, sys.argv[1])
import hdl_synth, paper_2609_36864_gb300 as hdl
for i, (n, d, V, dt) in enumerate([(700, 256, 9000, "bf16"), (300, 128, 4097, "f32"),
                                   (5, 64, 300, "bf16")]):
    spec = hdl_synth.small_spec("modes", n_roots=1, t_lo=n, t_hi=n, d=d, vocab=V, dtype=dt,
                                seed=40 + i)
    wl = hdl_synth.generate(spec, device="cuda")
    lp0, lp1, delta, ws = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets)
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
    np.save(sys.argv[2] + f"_{i}.npy", torch.stack([lp0, lp1, delta]).cpu().numpy())
"""


def test_rescore_cta_modes_agree_bitwise(hdl, tmp_path):
    """The two CTA organisations of the kernel (single CTA, cta_group::2
    pair) give bit-identical results, equal to the oracle's."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    outs = {}
    for mode in ("0", "2"):
        env = dict(os.environ, HDL_RESCORE_MODE=mode)
        stem = str(tmp_path / f"m{mode}")
        subprocess.run([sys.executable, "-c", _MODE_SCRIPT, root, stem], env=env, check=True,
                       timeout=300)
        outs[mode] = [np.load(stem + f"_{i}.npy") for i in range(3)]
    for i in range(3):
        assert np.array_equal(outs["0"][i], outs["2"][i], equal_nan=True)
    # and the shared result is the oracle's (first shape)
    spec = hdl_synth.small_spec("modes", n_roots=1, t_lo=700, t_hi=700, d=256, vocab=9000,
                                dtype="bf16", seed=40)
    wl = hdl_synth.generate(spec, device="cuda")
    W = to_f64(wl.w)
    y = wl.targets.cpu().numpy()
    assert_logp_close(outs["0"][0][0], oracle_logprobs(to_f64(wl.h_orig), W, y), "modes orig")
    assert_logp_close(outs["0"][0][1], oracle_logprobs(to_f64(wl.h_hind), W, y), "modes hind")


@pytest.mark.parametrize("n,d,V,dt", [(300, 256, 4097, "bf16"), (129, 128, 257, "bf16"),
                                      (1000, 1024, 8192, "bf16"), (200, 256, 5000, "f32"),
                                      (1, 64, 1, "bf16")])
def test_rescore_entropy(hdl, n, d, V, dt):
    """Next-token entropies of both contexts (the Entropy selector's signal,
    Section 4.1) against the oracle; asking for them leaves the log-probs
    unchanged bit for bit."""
    spec = hdl_synth.small_spec(f"e{n}_{d}_{V}", n_roots=1, t_lo=n, t_hi=n, d=d, vocab=V,
                                dtype=dt, seed=7 * n + V)
    wl = hdl_synth.generate(spec, device="cuda")
    lp0, lp1, de, e0, e1, ws = hdl.hdl_rescore_ex(wl.h_orig, wl.h_hind, wl.w, wl.targets,
                                                  want_entropy_hind=True)
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
    r = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets)
    assert torch.equal(lp0, r[0]) and torch.equal(lp1, r[1]) and torch.equal(de, r[2])
    import oracle
    W = to_f64(wl.w)
    h0, h1 = to_f64(wl.h_orig), to_f64(wl.h_hind)
    assert_logp_close(e0.cpu().numpy(), oracle.next_token_entropy(h0, W), "entropy orig")
    assert_logp_close(e1.cpu().numpy(), oracle.next_token_entropy(h1, W), "entropy hind")
    if V == 1:
        assert torch.all(e0.abs() < 1e-6)


def _tf32(x: np.ndarray, nearest: bool) -> np.ndarray:
    """fp32 -> tf32 (10 mantissa bits) as fp64: round to nearest even, or truncate."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    if nearest:
        b = b + 0xFFF + ((b >> 13) & 1)
    b = (b & 0xFFFFE000) & 0xFFFFFFFF
    return b.astype(np.uint32).view(np.float32).astype(np.float64)


def test_rescore_tf32_rounds_to_nearest(hdl):
    """fp32 inputs are rounded to tf32 to nearest (as the header states): the
    kernel matches the oracle on round-to-nearest tf32 inputs at fp32
    accumulation precision, and a truncating rounding is far from it."""
    spec = hdl_synth.small_spec("tf32rn", n_roots=1, t_lo=300, t_hi=300, d=512, vocab=3000,
                                dtype="f32", seed=77)
    wl = hdl_synth.generate(spec, device="cuda")
    lp0, lp1, _, ws = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets)
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
    got = lp0.cpu().numpy().astype(np.float64)
    h, w = wl.h_orig.cpu().numpy(), wl.w.cpu().numpy()
    y = wl.targets.cpu().numpy()
    err_rn = np.abs(got - oracle_logprobs(_tf32(h, True), _tf32(w, True), y)).max()
    err_tr = np.abs(got - oracle_logprobs(_tf32(h, False), _tf32(w, False), y)).max()
    assert err_rn < 5e-5, err_rn
    assert err_tr > 4 * err_rn, (err_tr, err_rn)


@pytest.mark.parametrize("V", [1, 257, 4096, 32000])
def test_rescore_zero_states_give_uniform(hdl, V):
    """All-zero hidden states: every logit is 0, so log p = -ln V for every
    token in both contexts and Delta = 0 (the closed form of a uniform
    distribution; V = 1 gives 0)."""
    n, d = 333, 128
    h = torch.zeros((n, d), dtype=torch.bfloat16, device="cuda")
    w = (torch.randn((V, d), device="cuda") * 0.02).to(torch.bfloat16)
    y = torch.randint(0, V, (n,), dtype=torch.int32, device="cuda")
    lp0, lp1, de, ws = hdl.hdl_rescore(h, h.clone(), w, y)
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
    ref = -np.log(V)
    assert np.all(np.abs(lp0.cpu().numpy() - ref) <= 1e-5 * max(1.0, abs(ref)))
    assert torch.equal(lp0, lp1) and torch.all(de == 0)


def test_rescore_large_logits(hdl):
    """Hidden states scaled 64x (logits in the hundreds, log-probs down to
    -10^3): the online max/sum stays finite and matches the oracle."""
    spec = hdl_synth.small_spec("big", n_roots=1, t_lo=400, t_hi=400, d=256, vocab=5000,
                                dtype="bf16", seed=91)
    wl = hdl_synth.generate(spec, device="cuda")
    h0 = (wl.h_orig.float() * 64).to(torch.bfloat16)
    h1 = (wl.h_hind.float() * 64).to(torch.bfloat16)
    lp0, lp1, de, ws = hdl.hdl_rescore(h0, h1, wl.w, wl.targets)
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
    W = to_f64(wl.w)
    y = wl.targets.cpu().numpy()
    r0 = oracle_logprobs(to_f64(h0), W, y)
    assert np.isfinite(lp0.cpu().numpy()).all() and r0.min() < -50
    assert_logp_close(lp0.cpu().numpy(), r0, "large orig")
    assert_logp_close(lp1.cpu().numpy(), oracle_logprobs(to_f64(h1), W, y), "large hind")


def test_rescore_concurrent_host_threads(hdl):
    """Two host threads, each on its own stream and workspace, calling the
    library at the same time: every result is bit-identical to the same call
    made alone (the library keeps no per-call state)."""
    import threading
    wls = [hdl_synth.generate(hdl_synth.small_spec(f"thr{i}", n_roots=2, t_lo=300, t_hi=500,
                                                   d=256, vocab=5000, seed=300 + i),
                              device="cuda") for i in range(2)]
    ref = []
    for wl in wls:
        lp0, lp1, de, _ = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets)
        bp, ns, bd = hdl.hdl_select_branches(de, wl.valid, wl.root_offsets, 8)
        ref.append((lp0, lp1, de, bp, ns))
    torch.cuda.synchronize()
    out = [None, None]
    errors = []

    def work(i):
        try:
            s = torch.cuda.Stream()
            wl = wls[i]
            res = []
            for _ in range(20):
                lp0, lp1, de, _ = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets,
                                                  stream=s)
                bp, ns, bd = hdl.hdl_select_branches(de, wl.valid, wl.root_offsets, 8, stream=s)
                res.append((lp0, lp1, de, bp, ns))
            s.synchronize()
            out[i] = res
        except Exception as e:   # surfaced below
            errors.append(e)

    ts = [threading.Thread(target=work, args=(i,)) for i in range(2)]
    for t in ts:
        t.start()
    for t in ts:
        t.join()
    assert not errors, errors
    for i in range(2):
        for res in out[i]:
            for a, b in zip(res, ref[i]):
                assert torch.equal(a, b)


@pytest.mark.parametrize("d,dt", [(8192, "bf16"), (16384, "bf16"), (8192, "f32")])
def test_rescore_wide_hidden(hdl, d, dt):
    """Hidden sizes of 70B-class models and beyond (long K loops: up to 256
    pipeline stages per tile) against the oracle."""
    spec = hdl_synth.small_spec(f"wide{d}{dt}", n_roots=1, t_lo=200, t_hi=200, d=d, vocab=1500,
                                dtype=dt, seed=d // 64)
    wl = hdl_synth.generate(spec, device="cuda")
    lp0, lp1, de, ws = hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets)
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
    W = to_f64(wl.w)
    y = wl.targets.cpu().numpy()
    assert_logp_close(lp0.cpu().numpy(), oracle_logprobs(to_f64(wl.h_orig), W, y), "wide orig")
    assert_logp_close(lp1.cpu().numpy(), oracle_logprobs(to_f64(wl.h_hind), W, y), "wide hind")


def test_rescore_randomized(hdl):
    """24 seeded random shapes (tokens 1-700, d a multiple of 64 up to 1024,
    vocabularies 1-10000, bf16 and fp32 states): log-probs, |Delta| and both
    entropies against the oracle element by element."""
    import oracle
    rng = np.random.default_rng(77)
    for case in range(24):
        n = int(rng.integers(1, 701))
        d = 64 * int(rng.integers(1, 17))
        V = int(rng.integers(1, 10001))
        dt = "f32" if case % 4 == 3 else "bf16"
        spec = hdl_synth.small_spec(f"rand{case}", n_roots=1, t_lo=n, t_hi=n, d=d, vocab=V,
                                    dtype=dt, seed=1000 + case)
        wl = hdl_synth.generate(spec, device="cuda")
        err, r0, r1, dl = run_and_check(hdl, wl, f"random case {case} {(n, d, V, dt)}")
        if case % 3 == 0:
            lp0, lp1, de, e0, e1, ws = hdl.hdl_rescore_ex(wl.h_orig, wl.h_hind, wl.w, wl.targets,
                                                          want_entropy_hind=True)
            assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
            W = to_f64(wl.w)
            assert_logp_close(e0.cpu().numpy(), oracle.next_token_entropy(to_f64(wl.h_orig), W),
                              f"random case {case} entropy orig")
            assert_logp_close(e1.cpu().numpy(), oracle.next_token_entropy(to_f64(wl.h_hind), W),
                              f"random case {case} entropy hind")
