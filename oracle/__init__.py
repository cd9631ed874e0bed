"""Plain CPU oracle for HDL re-scoring, branch selection and suffix masks.

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  The CUDA library
never calls it, and it shares no code with the CUDA library: it is a slow,
obviously correct restatement of the paper's definitions in float64 numpy,
so that the GPU results can be checked against it element by element.

Functions and the passages they follow (arXiv 2609.36864):
  target_logprobs        Section 3.1, Eq. (hindsight-contexts): log p_i(y_i)
                         under a softmax over the vocabulary at temperature 1
                         (the rollout temperature of Section 4.1).
  hindsight_divergence   Section 3.2, Eq. (div): s_i = |log p^H_i(y_i) - log p^0_i(y_i)|.
  next_token_entropy     Section 4.1 "Rollout protocols", the Entropy selector:
                         the entropy of the next-token distribution under the
                         original context, H = -sum_v p_v log p_v.
  select_branches        Section 3.2 (rank the candidate positions of a root by
                         s_i, take the highest), candidates = policy-generated
                         tokens (Section 3.1); optional spacing rule of
                         Section 4.4 (of points that sit too near each other,
                         one is kept).
  allocate_counts        Section 4.1 "Rollout protocols" (2 points, 3 + 4
                         continuations, G = 2 x (1 + 3 + 4) = 16), Table
                         (fork-ablation) 2x1 -> 7 and 4x2 -> 1 + 2, and
                         Section 4.4 (one point left: all continuations from it).
  assign_continuations   the same allocation, expanded per continuation.
  suffix_mask            Section 3.3: a root's loss covers its generated
                         tokens; a continuation's loss covers only the newly
                         sampled tokens y~_{>= i} of Eq. (branch-sampling).
  group_advantages       Section 3: A_j = R_j - mean of the group's rewards (no
                         standard-deviation normalisation, Section 4.1).
  grpo_token_loss        Section 4.1 "Training": the clipped policy objective
                         with asymmetric clipping (0.2 / 0.28), no KL term,
                         aggregated over tokens, on the suffix-only masks.

Readings where the paper is silent (each is also listed in the design notes):
  * ties in s_i go to the lower position;
  * fewer than k candidates: all of them are returned, the rest padded with -1;
  * NaN scores are not candidates;
  * the spacing rule takes min_gap (|t - a| < min_gap counts as too close) with two
    modes: greedy (walk the ranked list, skip a point too close to an accepted
    one) and drop-lower (take the plain top k, then drop each point too close
    to an accepted higher-ranked one);
  * allocation of C continuations over n points: point j of rank order gets
    floor(C / n) + [j < C mod n] (the extra ones to the higher-ranked points),
    or + [j >= n - C mod n] with ``extra_to_higher=False``;
  * the branch token itself is part of the sampled suffix (Eq. branch-sampling
    samples y~_{>= i}), so the mask includes position i; a continuation whose
    branch is -1 (its root had no candidate) gets an all-zero mask.

Parity pins: the tests in tests/test_oracle_pins.py check every function here
against brute force, closed forms, invariants and the paper's printed counts.
"""
from __future__ import annotations

import math

import numpy as np

__all__ = [
    "widen", "target_logprobs", "hindsight_divergence", "next_token_entropy",
    "select_branches",
    "allocate_counts", "assign_continuations", "suffix_mask", "group_advantages",
    "grpo_token_loss",
]


def widen(x, dtype: str) -> np.ndarray:
    """Exact float64 copy of an input array.

    ``dtype == "bf16"``: ``x`` holds the raw bf16 bit patterns (uint16/int16);
    a bf16 value is the upper half of an IEEE fp32, so shifting the pattern
    left by 16 bits gives the fp32 with the same value, widened exactly.
    ``dtype == "f32"``: ``x`` is float32 and is widened as-is.
    """
    x = np.asarray(x)
    if dtype == "bf16":
        bits = x.view(np.uint16).astype(np.uint32) << np.uint32(16)
        return bits.view(np.float32).astype(np.float64)
    if dtype == "f32":
        return x.astype(np.float32).astype(np.float64)
    raise ValueError(dtype)


def target_logprobs(h: np.ndarray, w: np.ndarray, targets: np.ndarray) -> np.ndarray:
    """log p(y_t) for every row of ``h`` (Eq. hindsight-contexts, Section 3.1).

    h: [n, d] float64 final-layer hidden states, w: [V, d] float64 LM head,
    targets: [n] ints in [0, V).  The next-token distribution is
    softmax(h W^T); its log at the target is z_y - log sum_v exp(z_v), taken
    with the row maximum subtracted first so that exp cannot overflow.
    """
    h = np.asarray(h, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)
    y = np.asarray(targets, dtype=np.int64)
    if h.shape[0] == 0:
        return np.zeros(0)
    z = h @ w.T                                         # logits [n, V]
    m = z.max(axis=1)
    log_norm = m + np.log(np.exp(z - m[:, None]).sum(axis=1))
    return z[np.arange(z.shape[0]), y] - log_norm


def hindsight_divergence(logp_hind: np.ndarray, logp_orig: np.ndarray) -> np.ndarray:
    """s_t = |log p^H_t(y_t) - log p^0_t(y_t)| (Eq. div, Section 3.2)."""
    return np.abs(np.asarray(logp_hind, np.float64) - np.asarray(logp_orig, np.float64))


def next_token_entropy(h: np.ndarray, w: np.ndarray) -> np.ndarray:
    """H_t = -sum_v p_v log p_v of p = softmax(h_t W^T), in nats (Section 4.1,
    the Entropy baseline's ranking signal).  log p_v is formed as
    z_v - max - log sum exp(z - max), so p_v = 0 contributes 0."""
    h = np.asarray(h, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)
    if h.shape[0] == 0:
        return np.zeros(0)
    z = h @ w.T
    m = z.max(axis=1, keepdims=True)
    logp = z - m - np.log(np.exp(z - m).sum(axis=1, keepdims=True))
    return -(np.exp(logp) * logp).sum(axis=1)


def _too_close(t: int, accepted: list, min_gap: int) -> bool:
    return any(abs(t - a) < min_gap for a in accepted)


def select_branches(delta, valid, root_offsets, k: int, min_gap: int = 0,
                    gap_mode: int = 0, lo: int = 0, hi: int = 0):
    """Top-k branch points per root (Section 3.2; spacing rule Section 4.4).

    delta: [N] scores; valid: [N] (nonzero = policy-generated) or None;
    root_offsets: [R + 1] packed root boundaries.  For each root the
    candidates are the positions t (relative to the root start) in
    [lo, hi) -- hi <= 0 meaning the root's end -- that are valid and whose
    score is not NaN.  They are ranked by score, descending, ties to the lower
    position, and the first k are taken (or the spacing rule applied).

    Returns (branch_pos [R, k] int32, -1 padded; n_selected [R] int32;
    branch_delta [R, k] float64, NaN padded), in rank order.
    """
    delta = np.asarray(delta, dtype=np.float64)
    offs = np.asarray(root_offsets, dtype=np.int64)
    R = len(offs) - 1
    pos = np.full((R, max(k, 0)), -1, dtype=np.int32)
    val = np.full((R, max(k, 0)), np.nan)
    nsel = np.zeros(R, dtype=np.int32)
    for r in range(R):
        start, end = int(offs[r]), int(offs[r + 1])
        T = end - start
        w_lo = max(lo, 0)
        w_hi = T if hi <= 0 else min(hi, T)
        cand = []
        for t in range(w_lo, w_hi):
            s = delta[start + t]
            if math.isnan(s):
                continue
            if valid is not None and not valid[start + t]:
                continue
            cand.append(t)
        ranked = sorted(cand, key=lambda t: (-delta[start + t], t))
        if min_gap <= 0:
            chosen = ranked[:k]
        else:
            pool = ranked if gap_mode == 0 else ranked[:k]
            chosen = []
            for t in pool:
                if len(chosen) == k:
                    break
                if not _too_close(t, chosen, min_gap):
                    chosen.append(t)
        nsel[r] = len(chosen)
        for j, t in enumerate(chosen):
            pos[r, j] = t
            val[r, j] = delta[start + t]
    return pos, nsel, val


def allocate_counts(n_points: int, n_conts: int, extra_to_higher: bool = True) -> list:
    """Continuations per branch point, in rank order (Section 4.1, Table fork-ablation).

    n_conts continuations are spread as evenly as possible over n_points
    points; the remainder goes to the higher-ranked points (or, with
    ``extra_to_higher=False``, to the lower-ranked ones).  One point left
    receives all of them (Section 4.4); no point left receives none.
    """
    if n_points <= 0:
        return []
    base, rem = divmod(n_conts, n_points)
    if extra_to_higher:
        return [base + (1 if j < rem else 0) for j in range(n_points)]
    return [base + (1 if j >= n_points - rem else 0) for j in range(n_points)]


def assign_continuations(n_selected, branch_pos, conts_per_root,
                         extra_to_higher: bool = True) -> np.ndarray:
    """Branch position (root-relative) of every continuation, root-major.

    Root r's conts_per_root[r] continuations follow those of roots < r; among
    them, the first count_0 branch from the rank-0 point, the next count_1 from
    the rank-1 point, and so on.  A root with no point gives -1.
    """
    out = []
    for r in range(len(conts_per_root)):
        n = int(n_selected[r])
        C = int(conts_per_root[r])
        if n == 0:
            out.extend([-1] * C)
            continue
        for j, cnt in enumerate(allocate_counts(n, C, extra_to_higher)):
            out.extend([int(branch_pos[r][j])] * cnt)
    return np.asarray(out, dtype=np.int32)


def suffix_mask(cont_branch, cont_offsets, cont_valid=None) -> np.ndarray:
    """Suffix-only loss mask of packed continuations (Section 3.3).

    Continuation c occupies [cont_offsets[c], cont_offsets[c+1]) and branched
    at root-relative position b = cont_branch[c]: token t of it carries loss
    iff t >= b and it is policy-generated.  b = 0 gives a root's mask (all of
    its generated tokens); b < 0 gives no loss at all.
    """
    offs = np.asarray(cont_offsets, dtype=np.int64)
    total = int(offs[-1]) if len(offs) else 0
    mask = np.zeros(total, dtype=np.uint8)
    for c in range(len(offs) - 1):
        b = int(cont_branch[c])
        start, end = int(offs[c]), int(offs[c + 1])
        if b < 0 or end <= start:
            continue
        t = np.arange(end - start)
        m = t >= b
        if cont_valid is not None:
            m &= np.asarray(cont_valid[start:end]) != 0
        mask[start:end] = m
    return mask


def group_advantages(rewards, group_offsets) -> np.ndarray:
    """A_j = R_j - (1/G) sum_{k in group} R_k for every trajectory (Section 3).

    Group g holds trajectories [group_offsets[g], group_offsets[g+1]) -- its
    roots and their continuations (Section 3.3: they form one group).
    """
    R = np.asarray(rewards, dtype=np.float64)
    offs = np.asarray(group_offsets, dtype=np.int64)
    A = np.zeros(len(R))
    for g in range(len(offs) - 1):
        lo, hi = int(offs[g]), int(offs[g + 1])
        if hi > lo:
            A[lo:hi] = R[lo:hi] - R[lo:hi].mean()
    return A


def grpo_token_loss(logp_new, logp_old, mask, traj_offsets, advantages,
                    eps_low: float = 0.2, eps_high: float = 0.28):
    """Clipped policy loss aggregated over tokens (Section 4.1).

    For token t of trajectory j with mask m_t (Section 3.3's suffix-only mask):
      r_t   = exp(logp_new_t - logp_old_t)
      obj_t = min(r_t A_j, clip(r_t, 1 - eps_low, 1 + eps_high) A_j)
      loss  = - sum_t m_t obj_t / sum_t m_t
    and grad_t = d loss / d logp_new_t, which is -m_t r_t A_j / sum m when the
    unclipped term is the minimum (ties included) and 0 otherwise.  Every
    quantity, the choice of the minimum included, is taken in float64.
    Returns (loss, grad, stats) with stats = (masked tokens, fraction of masked
    tokens whose clipped term is strictly the minimum, mean masked ratio).
    """
    lpn = np.asarray(logp_new, dtype=np.float64)
    lpo = np.asarray(logp_old, dtype=np.float64)
    m = np.asarray(mask) != 0
    offs = np.asarray(traj_offsets, dtype=np.int64)
    A = np.zeros(len(lpn))
    for j in range(len(offs) - 1):
        A[int(offs[j]):int(offs[j + 1])] = advantages[j]
    r = np.exp(lpn - lpo)
    unclipped = r * A
    clipped = np.clip(r, 1.0 - eps_low, 1.0 + eps_high) * A
    n = int(m.sum())
    if n == 0:
        return 0.0, np.zeros(len(lpn)), (0, 0.0, 0.0)
    active = unclipped <= clipped            # the unclipped term is the minimum
    obj = np.where(active, unclipped, clipped)
    loss = -obj[m].sum() / n
    grad = np.where(m & active, -r * A / n, 0.0)
    clip_frac = float((~active[m]).sum()) / n
    return float(loss), grad, (n, clip_frac, float(r[m].mean()))
