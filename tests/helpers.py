"""Bridges between the generated workloads, the CPU oracle and the tolerances
of the parity tests (test code: the library never imports this)."""
from __future__ import annotations

import numpy as np
import torch

import oracle

# Log-probability tolerance: |err| <= ATOL + RTOL * |ref|.
LP_ATOL = 1e-3
LP_RTOL = 1e-3
# End-to-end selection may differ only at positions whose reference score is
# within this band of the root's k-th selected score.
SELECT_BAND = 2e-3


def to_f64(t: torch.Tensor) -> np.ndarray:
    """Exact float64 copy of a bf16 or fp32 tensor (via the oracle's widening)."""
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return oracle.widen(t.view(torch.int16).numpy(), "bf16")
    if t.dtype == torch.float32:
        return oracle.widen(t.numpy(), "f32")
    raise TypeError(t.dtype)


def oracle_logprobs(h64: np.ndarray, w64: np.ndarray, y: np.ndarray, block: int = 1024):
    """oracle.target_logprobs over row blocks (each row is independent)."""
    out = np.empty(h64.shape[0])
    for s in range(0, h64.shape[0], block):
        out[s:s + block] = oracle.target_logprobs(h64[s:s + block], w64, y[s:s + block])
    return out


def assert_logp_close(got, ref, what=""):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    err = np.abs(got - ref)
    bound = LP_ATOL + LP_RTOL * np.abs(ref)
    bad = ~(err <= bound)
    assert not bad.any(), (f"{what}: {bad.sum()} of {bad.size} outside tolerance; "
                           f"max err {err.max():.3e} at {int(err.argmax())}")
    return float(err.max()) if err.size else 0.0


def sample_rows(n: int, count: int, seed: int = 0) -> np.ndarray:
    """First, last and random rows (sorted, unique)."""
    rng = np.random.default_rng(seed)
    pick = set([0, n - 1]) | set(rng.integers(0, n, size=count).tolist())
    return np.array(sorted(pick), dtype=np.int64)


def check_selection_band(gpu_pos, gpu_nsel, ref_delta, valid, offs, k, band=SELECT_BAND):
    """GPU branch sets vs. the oracle's on the oracle's scores: equal except at
    positions whose reference score lies within ``band`` of the k-th value."""
    pos, nsel, _ = oracle.select_branches(ref_delta, valid, offs, k)
    gpu_pos = np.asarray(gpu_pos)
    for r in range(len(offs) - 1):
        assert int(gpu_nsel[r]) == int(nsel[r]), (r, gpu_nsel[r], nsel[r])
        n = int(nsel[r])
        if n == 0:
            continue
        a = set(gpu_pos[r, :n].tolist())
        b = set(pos[r, :n].tolist())
        kth = ref_delta[offs[r] + pos[r, n - 1]]
        for t in a ^ b:
            assert abs(ref_delta[offs[r] + t] - kth) <= band, (r, t, ref_delta[offs[r] + t], kth)


# GRPO: tokens closer than this many float32 ulps to a clip bound may be
# decided either way by a float32 kernel (the float32 difference of the
# log-probs is rounded, and CUDA's expf may differ from the exact ratio by
# up to 2 ulp), so the float64 oracle's decision is not binding there.
GRPO_DECISION_ULPS = 4


def grpo_decided(lpn, lpo, eps_low=0.2, eps_high=0.28):
    """Tokens whose ratio exp(lpn - lpo), taken in float64, lies more than
    GRPO_DECISION_ULPS float32 ulps from 1 - eps_low and 1 + eps_high: there
    a float32 kernel and the float64 oracle must pick the same term."""
    r = np.exp(np.asarray(lpn, np.float64) - np.asarray(lpo, np.float64))
    ok = np.ones(len(r), dtype=bool)
    for b in (1.0 - eps_low, 1.0 + eps_high):
        ok &= np.abs(r - b) > GRPO_DECISION_ULPS * float(np.spacing(np.float32(b)))
    return ok


def check_grpo(adv, grad, stats, lpn, lpo, mask, toffs, rewards, goffs, grad_slice=None):
    """The GRPO update's outputs (host arrays) against the oracle, which
    takes only the inputs: advantages within 1e-6, loss 1e-5 relative,
    gradient 1e-5 of its largest entry on the tokens both sides must decide
    alike; the clip fraction may differ by the undecided masked tokens."""
    A_ref = oracle.group_advantages(rewards, goffs)
    assert np.allclose(adv, A_ref, rtol=0, atol=1e-6), np.abs(adv - A_ref).max()
    loss, g_ref, (n, clip_frac, mean_r) = oracle.grpo_token_loss(lpn, lpo, mask, toffs, A_ref)
    assert stats[1] == n
    assert abs(stats[0] - loss) <= 1e-5 * max(1.0, abs(loss)), (stats[0], loss)
    ok = grpo_decided(lpn, lpo)
    m = np.asarray(mask) != 0
    undecided = int((m & ~ok).sum())
    assert abs(stats[2] - clip_frac) <= 1e-6 + undecided / max(n, 1), (stats[2], clip_frac)
    assert abs(stats[3] - mean_r) <= 1e-5
    g = grad if grad_slice is None else grad[grad_slice]
    tol = 1e-5 * np.abs(g_ref).max() if g_ref.size else 0.0
    assert np.all((g == 0)[ok] == (g_ref == 0)[ok])
    assert np.all(np.abs(g - g_ref)[ok] <= tol)
    assert np.all(g[~m] == 0)
    # near a bound either term may be the minimum: the gradient there is the
    # unclipped one, -r A / n, or 0, and nothing else
    amb = m & ~ok
    if amb.any():
        r = np.exp(np.asarray(lpn, np.float64) - np.asarray(lpo, np.float64))
        A = np.repeat(A_ref, np.diff(np.asarray(toffs, np.int64)))
        unclipped = -r * A / n
        dev = np.minimum(np.abs(g - unclipped), np.abs(g))[amb]
        assert np.all(dev <= tol), dev.max()
    return undecided
