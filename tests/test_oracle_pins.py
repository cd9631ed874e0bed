"""Pins for the CPU oracle: it is checked against things other than itself.

Each ``check_*`` function takes the implementation under test as an argument,
so the same check runs on the oracle (must pass) and on deliberately broken
copies of it (``test_planted_mistakes_*``: must fail).  The pins are
  * brute force from the textbook definitions (pure-Python fsum softmax,
    enumeration of all subsets for the top-k and spacing rules),
  * closed forms (uniform logits, two-word and one-word vocabularies),
  * invariants (normalisation, shift invariance, Delta = 0 for identical
    contexts, symmetry),
  * a library routine for the ranking (numpy.lexsort) and torch's exact bf16
    widening,
  * the counts the paper prints for its branching configurations.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------- log-probs
def brute_logp(h, w, y):
    """log p(y) = log( e^{z_y} / sum_v e^{z_v} ), z_v = <h, w_v>, in fsum."""
    z = [math.fsum(a * b for a, b in zip(h, wv)) for wv in w]
    den = math.fsum(math.exp(v) for v in z)
    return math.log(math.exp(z[y]) / den)


def check_logp_bruteforce(fn):
    rng = np.random.default_rng(7)
    for d, V in [(1, 1), (1, 2), (3, 5), (4, 8), (2, 7)]:
        h = rng.normal(size=(6, d))
        w = rng.normal(size=(V, d))
        y = rng.integers(0, V, size=6)
        got = fn(h, w, y)
        ref = [brute_logp(h[i], w, int(y[i])) for i in range(6)]
        assert np.allclose(got, ref, rtol=0, atol=1e-12), (d, V, got, ref)


def check_logp_closed_forms(fn):
    # uniform logits (W = 0): log p = -ln V for every target
    for V in (1, 2, 3, 4096):
        got = fn(np.ones((3, 4)), np.zeros((V, 4)), np.array([0, V - 1, V // 2]))
        assert np.allclose(got, -math.log(V), rtol=0, atol=1e-14), (V, got)
    # V = 2, d = 1: z = (a b0, a b1): log p(0) = -log1p(exp(z1 - z0))
    a, b0, b1 = 1.7, 0.9, -2.3
    got = fn(np.array([[a]]), np.array([[b0], [b1]]), np.array([0]))
    assert abs(got[0] + math.log1p(math.exp(a * b1 - a * b0))) < 1e-15
    got = fn(np.array([[a]]), np.array([[b0], [b1]]), np.array([1]))
    assert abs(got[0] + math.log1p(math.exp(a * b0 - a * b1))) < 1e-15
    # a single-word vocabulary is certain
    assert fn(np.array([[5.0, -1.0]]), np.array([[0.3, 0.2]]), np.array([0]))[0] == 0.0
    # the target column is the one gathered: logits (0, 10, 0, 0)
    w = np.array([[0.0], [10.0], [0.0], [0.0]])
    got = fn(np.array([[1.0], [1.0]]), w, np.array([1, 2]))
    assert abs(got[0] - (10 - math.log(math.exp(10) + 3))) < 1e-13
    assert abs(got[1] - (0 - math.log(math.exp(10) + 3))) < 1e-13


def check_logp_normalised(fn):
    rng = np.random.default_rng(3)
    d, V = 16, 300
    h = rng.normal(size=(1, d)) * 3
    w = rng.normal(size=(V, d))
    lp = fn(np.repeat(h, V, axis=0), w, np.arange(V))
    assert np.all(lp <= 0)
    assert abs(math.fsum(np.exp(lp)) - 1.0) < 1e-12


def check_logp_shift_invariant(fn):
    # append a constant feature: all logits move by c = 800, log p must not
    # change (and must stay finite: exp(800) overflows without the max shift)
    rng = np.random.default_rng(5)
    h = rng.normal(size=(4, 8))
    w = rng.normal(size=(50, 8))
    y = rng.integers(0, 50, size=4)
    base = fn(h, w, y)
    h2 = np.concatenate([h, np.ones((4, 1))], axis=1)
    w2 = np.concatenate([w, np.full((50, 1), 800.0)], axis=1)
    shifted = fn(h2, w2, y)
    assert np.all(np.isfinite(shifted))
    assert np.allclose(base, shifted, rtol=0, atol=1e-10)


def test_logp_bruteforce():
    check_logp_bruteforce(O.target_logprobs)


def test_logp_closed_forms():
    check_logp_closed_forms(O.target_logprobs)


def test_logp_normalised():
    check_logp_normalised(O.target_logprobs)


def test_logp_shift_invariant():
    check_logp_shift_invariant(O.target_logprobs)


def test_logp_empty():
    assert O.target_logprobs(np.zeros((0, 4)), np.ones((3, 4)), np.zeros(0, int)).shape == (0,)


def test_widen_bf16_exact():
    pats = {0x3F80: 1.0, 0xC000: -2.0, 0x3F81: 1.0 + 2.0 ** -7, 0x0001: 2.0 ** -133,
            0x7F7F: (2 - 2.0 ** -7) * 2.0 ** 127, 0x8000: -0.0, 0x0000: 0.0}
    bits = np.array(list(pats.keys()), dtype=np.uint16)
    got = O.widen(bits, "bf16")
    assert list(got) == list(pats.values())
    # torch's bf16 -> fp32 conversion is exact: both must agree on random values
    t = (torch.randn(10000, generator=torch.Generator().manual_seed(1)) * 50).to(torch.bfloat16)
    ref = t.float().double().numpy()
    assert np.array_equal(O.widen(t.view(torch.int16).numpy(), "bf16"), ref)
    f = np.array([1.5, -3.25e-7, 1e30], dtype=np.float32)
    assert np.array_equal(O.widen(f, "f32"), f.astype(np.float64))


# ---------------------------------------------------------------- divergence
def check_divergence(fn):
    rng = np.random.default_rng(11)
    h = rng.normal(size=(20, 6))
    w = rng.normal(size=(30, 6))
    y = rng.integers(0, 30, size=20)
    lp = O.target_logprobs(h, w, y)
    assert np.all(fn(lp, lp) == 0.0)                       # identical contexts
    lp2 = O.target_logprobs(h + rng.normal(size=h.shape), w, y)
    a, b = fn(lp2, lp), fn(lp, lp2)
    assert np.array_equal(a, b)                              # symmetric
    assert np.all(a >= 0)
    assert fn(np.array([-1.0]), np.array([-3.0]))[0] == 2.0   # |(-1) - (-3)|
    assert fn(np.array([-3.0]), np.array([-1.0]))[0] == 2.0


def test_divergence():
    check_divergence(O.hindsight_divergence)


# ------------------------------------------------------------------ entropy
def brute_entropy(h, w):
    z = [math.fsum(a * b for a, b in zip(h, wv)) for wv in w]
    den = math.fsum(math.exp(v) for v in z)
    p = [math.exp(v) / den for v in z]
    return -math.fsum(q * math.log(q) for q in p if q > 0)


def check_entropy(fn):
    rng = np.random.default_rng(13)
    for d, V in [(1, 1), (1, 2), (3, 5), (4, 8)]:
        h = rng.normal(size=(5, d))
        w = rng.normal(size=(V, d))
        got = fn(h, w)
        ref = [brute_entropy(h[i], w) for i in range(5)]
        assert np.allclose(got, ref, rtol=0, atol=1e-12), (d, V, got, ref)
    # uniform logits: ln V; V = 1: 0
    for V in (1, 2, 7, 4096):
        assert np.allclose(fn(np.ones((2, 3)), np.zeros((V, 3))), math.log(V), atol=1e-13)
    # two words: the binary entropy of sigmoid(z0 - z1)
    a, b0, b1 = 0.7, 2.0, -1.0
    p0 = 1.0 / (1.0 + math.exp(a * b1 - a * b0))
    hb = -p0 * math.log(p0) - (1 - p0) * math.log(1 - p0)
    assert abs(fn(np.array([[a]]), np.array([[b0], [b1]]))[0] - hb) < 1e-15
    # one dominant word: ~0; bounds 0 <= H <= ln V; shift and permutation invariance
    w = np.zeros((50, 2))
    w[3, 0] = 60.0
    assert 0 <= fn(np.array([[1.0, 0.0]]), w)[0] < 1e-20
    h = rng.normal(size=(6, 8))
    w = rng.normal(size=(40, 8))
    H = fn(h, w)
    assert np.all(H >= 0) and np.all(H <= math.log(40) + 1e-12)
    h2 = np.concatenate([h, np.ones((6, 1))], axis=1)
    w2 = np.concatenate([w, np.full((40, 1), 700.0)], axis=1)
    assert np.allclose(fn(h2, w2), H, atol=1e-10)
    assert np.allclose(fn(h, w[rng.permutation(40)]), H, atol=1e-12)


def test_entropy():
    check_entropy(O.next_token_entropy)


def test_planted_mistakes_entropy():
    def no_minus(h, w):
        return -O.next_token_entropy(h, w)

    def log2_units(h, w):
        return O.next_token_entropy(h, w) / math.log(2)

    def unnormalised(h, w):
        z = np.asarray(h, float) @ np.asarray(w, float).T
        e = np.exp(z - z.max(1, keepdims=True))
        return -(e * np.log(e)).sum(1)
    for mutant in (no_minus, log2_units, unnormalised):
        with pytest.raises(AssertionError):
            check_entropy(mutant)


# ----------------------------------------------------------------- selection
def _beats(delta, a, b):
    return delta[a] > delta[b] or (delta[a] == delta[b] and a < b)


def brute_select(delta, valid, T, k, min_gap=0, gap_mode=0, lo=0, hi=0):
    """Enumerate subsets: the unique top-m set, or the lexicographically best
    spacing-feasible set (best = lowest rank at the first difference, and a
    set beats any of its prefixes)."""
    w_hi = T if hi <= 0 else min(hi, T)
    cand = [t for t in range(max(lo, 0), w_hi)
            if not math.isnan(delta[t]) and (valid is None or valid[t])]
    rank = {t: sum(_beats(delta, c, t) for c in cand) for t in cand}
    m = min(k, len(cand))
    tops = [S for S in itertools.combinations(cand, m)
            if all(_beats(delta, s, c) for s in S for c in cand if c not in S)]
    assert len(tops) == 1
    top = sorted(tops[0], key=lambda t: rank[t])
    if min_gap <= 0:
        return top
    pool = cand if gap_mode == 0 else top
    best, best_key = [], None
    for size in range(0, min(k, len(pool)) + 1):
        for S in itertools.combinations(pool, size):
            if any(abs(a - b) < min_gap for a, b in itertools.combinations(S, 2)):
                continue
            key = tuple(sorted(rank[t] for t in S)) + (math.inf,) * (k - size)
            if best_key is None or key < best_key:
                best, best_key = S, key
    return sorted(best, key=lambda t: rank[t])


def _random_select_case(rng):
    T = int(rng.integers(0, 11))
    delta = rng.integers(0, 4, size=T) * 0.5          # many ties
    if T and rng.random() < 0.3:
        delta[rng.integers(0, T)] = np.nan
    valid = (rng.random(T) < 0.8).astype(np.uint8) if rng.random() < 0.7 else None
    k = int(rng.integers(0, 6))
    lo = int(rng.integers(0, 3)) if rng.random() < 0.3 else 0
    hi = int(rng.integers(0, T + 2)) if rng.random() < 0.3 else 0
    return delta, valid, T, k, lo, hi


def check_select_bruteforce(fn, n_cases=300, gap=False):
    rng = np.random.default_rng(2024 + gap)
    for _ in range(n_cases):
        delta, valid, T, k, lo, hi = _random_select_case(rng)
        mg = int(rng.integers(1, 4)) if gap else 0
        mode = int(rng.integers(0, 2)) if gap else 0
        pos, nsel, val = fn(delta, valid, [0, T], k, min_gap=mg, gap_mode=mode, lo=lo, hi=hi)
        ref = brute_select(delta, valid, T, k, mg, mode, lo, hi)
        assert nsel[0] == len(ref), (delta, valid, k, mg, mode, lo, hi, pos, ref)
        assert list(pos[0, :len(ref)]) == ref, (delta, valid, k, mg, mode, lo, hi, pos, ref)
        assert np.all(pos[0, len(ref):] == -1)
        assert np.array_equal(val[0, :len(ref)], delta[ref]) if ref else True
        assert np.all(np.isnan(val[0, len(ref):]))


def test_select_bruteforce():
    check_select_bruteforce(O.select_branches)


def test_select_gap_bruteforce():
    check_select_bruteforce(O.select_branches, gap=True)


def test_select_vs_lexsort():
    """Plain top-k equals numpy.lexsort over (-delta, t) among candidates."""
    rng = np.random.default_rng(9)
    lengths = [0, 1, 5, 17, 700, 4096, 3000]
    offs = np.concatenate([[0], np.cumsum(lengths)])
    N = int(offs[-1])
    delta = np.round(rng.exponential(size=N), 2).astype(np.float32).astype(np.float64)
    valid = (rng.random(N) < 0.8).astype(np.uint8)
    for k in (1, 8, 16):
        pos, nsel, val = O.select_branches(delta, valid, offs, k)
        for r in range(len(lengths)):
            s, e = offs[r], offs[r + 1]
            t = np.arange(e - s)
            c = t[valid[s:e] != 0]
            order = c[np.lexsort((c, -delta[s:e][c]))][:k]
            assert nsel[r] == len(order)
            assert np.array_equal(pos[r, :len(order)], order)


# ---------------------------------------------------------------- allocation
def test_allocation_paper_counts():
    g = json.load(open(os.path.join(GOLDEN, "allocation_paper.json")))
    for cfg in g["configs"]:
        counts = O.allocate_counts(cfg["points_per_root"], cfg["conts_per_root"])
        assert sorted(counts) == sorted(cfg["counts"]), cfg
        assert cfg["roots"] * (1 + sum(counts)) == cfg["group_size"]
        assert cfg["roots"] * len(counts) == cfg["max_points_per_group"]
        flipped = O.allocate_counts(cfg["points_per_root"], cfg["conts_per_root"], False)
        assert sorted(flipped) == sorted(cfg["counts"])
    one = g["one_point_left"]
    assert O.allocate_counts(one["points_selected"], one["conts_per_root"]) == one["counts"]


def test_allocation_rank_order():
    # the extra continuation goes to the higher-ranked point (or the lower)
    assert O.allocate_counts(2, 7) == [4, 3]
    assert O.allocate_counts(2, 7, extra_to_higher=False) == [3, 4]
    assert O.allocate_counts(3, 8) == [3, 3, 2]
    assert O.allocate_counts(3, 8, extra_to_higher=False) == [2, 3, 3]
    assert O.allocate_counts(4, 2) == [1, 1, 0, 0]
    assert O.allocate_counts(0, 5) == []
    for n in range(1, 9):
        for C in range(0, 20):
            c = O.allocate_counts(n, C)
            assert sum(c) == C and max(c) - min(c) <= 1


def test_assign_layout():
    bp = np.array([[5, 9, -1], [2, -1, -1], [-1, -1, -1]])
    got = O.assign_continuations([2, 1, 0], bp, [7, 3, 2])
    assert got.tolist() == [5, 5, 5, 5, 9, 9, 9, 2, 2, 2, -1, -1]


# ---------------------------------------------------------------------- mask
def check_mask(fn):
    rng = np.random.default_rng(4)
    lens = [0, 1, 7, 33, 64, 129]
    offs = np.concatenate([[0], np.cumsum(lens)])
    valid = (rng.random(int(offs[-1])) < 0.7).astype(np.uint8)
    for b in (0, 1, 6, 32, 200, -1):
        br = np.full(len(lens), b)
        m = fn(br, offs, valid)
        for c, L in enumerate(lens):
            s = int(offs[c])
            seg = m[s:s + L]
            for t in range(L):                       # element by element
                want = 1 if (b >= 0 and t >= b and valid[s + t]) else 0
                assert seg[t] == want
            if b >= 0:
                assert int(seg.sum()) == int(valid[s + max(b, 0):s + L].sum())
    # b = 0 reproduces a root's mask (its policy-generated tokens)
    assert np.array_equal(fn(np.zeros(len(lens), int), offs, valid), valid)
    # no validity mask: every token at or after b
    m = fn(np.array([3]), np.array([0, 10]), None)
    assert m.tolist() == [0, 0, 0] + [1] * 7


def test_mask():
    check_mask(O.suffix_mask)


# ------------------------------------------------- planted mistakes must fail
def _lp_no_max_shift(h, w, y):
    z = np.asarray(h, float) @ np.asarray(w, float).T
    return z[np.arange(len(z)), y] - np.log(np.exp(z).sum(1))


def _lp_off_by_one(h, w, y):
    y = (np.asarray(y) + 1) % np.asarray(w).shape[0]
    return O.target_logprobs(h, w, y)


def _lp_no_log(h, w, y):
    z = np.asarray(h, float) @ np.asarray(w, float).T
    m = z.max(1)
    return z[np.arange(len(z)), y] - m - np.exp(z - m[:, None]).sum(1)


def _lp_transposed(h, w, y):
    z = np.asarray(h, float) @ np.asarray(w, float).T
    z = z - z.mean(0, keepdims=True)          # normalises over the wrong axis
    m = z.max(1)
    return z[np.arange(len(z)), y] - m - np.log(np.exp(z - m[:, None]).sum(1))


@pytest.mark.parametrize("mutant", [_lp_no_max_shift, _lp_off_by_one, _lp_no_log, _lp_transposed])
def test_planted_mistakes_logp(mutant):
    failed = 0
    for chk in (check_logp_bruteforce, check_logp_closed_forms,
                check_logp_normalised, check_logp_shift_invariant):
        try:
            with np.errstate(all="ignore"):
                chk(mutant)
        except (AssertionError, IndexError, ValueError):
            failed += 1
    assert failed >= 1


def test_planted_mistakes_divergence():
    for mutant in (lambda a, b: np.asarray(a) - np.asarray(b),
                   lambda a, b: np.abs(np.asarray(a)) - np.abs(np.asarray(b))):
        with pytest.raises(AssertionError):
            check_divergence(mutant)


def _sel_ties_high(delta, valid, offs, k, min_gap=0, gap_mode=0, lo=0, hi=0):
    # ranks ties to the higher position
    T = int(offs[1])
    w_hi = T if hi <= 0 else min(hi, T)
    cand = [t for t in range(max(lo, 0), w_hi)
            if not math.isnan(delta[t]) and (valid is None or valid[t])]
    chosen = sorted(cand, key=lambda t: (-delta[t], -t))[:k]
    pos = np.full((1, k), -1, np.int32)
    val = np.full((1, k), np.nan)
    pos[0, :len(chosen)] = chosen
    val[0, :len(chosen)] = [delta[t] for t in chosen]
    return pos, np.array([len(chosen)], np.int32), val


def _sel_ignores_valid(delta, valid, offs, k, **kw):
    return O.select_branches(delta, None, offs, k, **kw)


def _sel_gap_inclusive(delta, valid, offs, k, min_gap=0, **kw):
    return O.select_branches(delta, valid, offs, k, min_gap=max(min_gap - 1, 0), **kw)


def test_planted_mistakes_select():
    for mutant, gap in ((_sel_ties_high, False), (_sel_ignores_valid, False),
                        (_sel_gap_inclusive, True)):
        with pytest.raises(AssertionError):
            check_select_bruteforce(mutant, gap=gap)


def test_planted_mistakes_mask():
    def strict(br, offs, valid):             # t > b instead of t >= b
        return O.suffix_mask(np.asarray(br) + np.where(np.asarray(br) >= 0, 1, 0), offs, valid)

    def ignores_valid(br, offs, valid):
        return O.suffix_mask(br, offs, None)
    for mutant in (strict, ignores_valid):
        with pytest.raises(AssertionError):
            check_mask(mutant)



# ------------------------------------------------------- GRPO update (next)
def check_advantages(fn):
    A = fn([1.0, 0.0, 0.5, 0.5, 3.0, 2.0, 2.0, 2.0], [0, 3, 5, 5, 8])
    assert np.allclose(A, [0.5, -0.5, 0.0, -1.25, 1.25, 0.0, 0.0, 0.0], atol=1e-15)
    rng = np.random.default_rng(1)
    offs = np.concatenate([[0], np.cumsum(rng.integers(1, 17, size=20))])
    R = rng.random(offs[-1])
    A = fn(R, offs)
    for g in range(20):
        assert abs(A[offs[g]:offs[g + 1]].sum()) < 1e-12      # mean-centred
    assert np.all(fn(np.ones(16), [0, 16]) == 0)              # uniform rewards: no signal


def test_advantages():
    check_advantages(O.group_advantages)


def check_grpo_loss(fn):
    # hand cases of the asymmetric clip (eps 0.2 / 0.28), one token each:
    # (ratio, advantage, objective, gradient d loss / d logp_new, clipped?)
    # -- the gradient is -r A where the unclipped term is the minimum (ties
    # included: inside [0.8, 1.28] both terms are equal) and 0 where the
    # clipped term is strictly smaller
    for r, A, want, want_g, want_clip in (
            (1.5, 1.0, 1.28, 0.0, 1), (0.5, -1.0, -0.8, 0.0, 1), (0.5, 1.0, 0.5, -0.5, 0),
            (1.5, -1.0, -1.5, 1.5, 0), (1.1, 2.0, 2.2, -2.2, 0), (0.7, 1.0, 0.7, -0.7, 0),
            (1.0, -3.0, -3.0, 3.0, 0)):
        loss, grad, st = fn([math.log(r)], [0.0], [1], [0, 1], [A])
        assert abs(loss + want) < 1e-12, (r, A, loss)
        assert abs(grad[0] - want_g) < 1e-12, (r, A, grad[0])
        assert st[0] == 1 and st[1] == want_clip and abs(st[2] - r) < 1e-12, (r, A, st)
    # ratio 1: loss = -sum_j A_j L_j / sum_j L_j over masked tokens
    offs = [0, 3, 7, 8]
    mask = [1, 1, 0, 1, 1, 1, 1, 0]
    A = [1.0, -0.5, 2.0]
    loss, grad, st = fn(np.zeros(8), np.zeros(8), mask, offs, A)
    assert abs(loss - (-(1.0 * 2 + (-0.5) * 4) / 6)) < 1e-12 and st[0] == 6
    assert grad[2] == 0 and grad[7] == 0                       # masked tokens carry none
    # gradient = central finite difference of the loss (away from clip edges)
    rng = np.random.default_rng(2)
    n = 40
    offs = [0, 10, 25, 40]
    A = [0.7, -1.3, 0.4]
    lpo = rng.normal(size=n)
    lpn = lpo + rng.uniform(-0.5, 0.5, size=n)
    mask = (rng.random(n) < 0.8).astype(np.uint8)
    loss, grad, _ = fn(lpn, lpo, mask, offs, A)
    h = 1e-6
    for t in range(n):
        e = np.zeros(n)
        e[t] = h
        lp = fn(lpn + e, lpo, mask, offs, A)[0]
        lm = fn(lpn - e, lpo, mask, offs, A)[0]
        fd = (lp - lm) / (2 * h)
        r = math.exp(lpn[t] - lpo[t])
        if abs(r - 0.8) > 1e-3 and abs(r - 1.28) > 1e-3:
            assert abs(fd - grad[t]) < 1e-7, (t, fd, grad[t])
    # masked tokens do not move the loss
    lpn2 = lpn.copy()
    lpn2[mask == 0] += 3.0
    assert abs(fn(lpn2, lpo, mask, offs, A)[0] - loss) < 1e-15


def test_grpo_loss():
    check_grpo_loss(O.grpo_token_loss)


def test_planted_mistakes_grpo():
    def std_normalised(R, offs):
        A = O.group_advantages(R, offs)
        R = np.asarray(R, float)
        for g in range(len(offs) - 1):
            if offs[g + 1] <= offs[g]:
                continue
            sd = R[offs[g]:offs[g + 1]].std()
            if sd > 0:
                A[offs[g]:offs[g + 1]] /= sd
        return A
    with pytest.raises(AssertionError):
        check_advantages(std_normalised)

    def symmetric_clip(lpn, lpo, mask, offs, A):
        return O.grpo_token_loss(lpn, lpo, mask, offs, A, 0.2, 0.2)

    def sequence_mean(lpn, lpo, mask, offs, A):
        loss, grad, st = O.grpo_token_loss(lpn, lpo, mask, offs, A)
        m = np.asarray(mask) != 0
        per = []
        for j in range(len(offs) - 1):
            s_, e_ = offs[j], offs[j + 1]
            if m[s_:e_].any():
                l_, _, _ = O.grpo_token_loss(lpn[s_:e_], lpo[s_:e_], mask[s_:e_],
                                             [0, e_ - s_], [A[j]])
                per.append(l_)
        return float(np.mean(per)), grad, st

    def no_clip(lpn, lpo, mask, offs, A):
        return O.grpo_token_loss(lpn, lpo, mask, offs, A, 1e9, 1e9)

    def ties_to_clipped(lpn, lpo, mask, offs, A):
        # the gradient taken from the clipped term whenever it is not larger
        loss, grad, st = O.grpo_token_loss(lpn, lpo, mask, offs, A)
        r = np.exp(np.asarray(lpn, float) - np.asarray(lpo, float))
        Aj = np.repeat(np.asarray(A, float), np.diff(offs))
        tie = np.isclose(r * Aj, np.clip(r, 0.8, 1.28) * Aj, rtol=0, atol=0)
        return loss, np.where(tie, 0.0, grad), st
    for mutant in (symmetric_clip, sequence_mean, no_clip, ties_to_clipped):
        with pytest.raises(AssertionError):
            check_grpo_loss(mutant)
