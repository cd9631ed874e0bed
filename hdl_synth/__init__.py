"""Seeded synthetic inputs for HDL hindsight re-scoring and branch selection.

This module only draws random inputs; it holds none of the method's arithmetic
(no log-softmax, no divergence, no selection, no masks).  Both the CPU oracle
(via the tests and the bench) and the CUDA path consume the tensors it returns,
which is the only thing the two sides share.

What is modelled (Section 3 of the paper): one problem's root trajectories
y = (y_1..y_T), the final-layer hidden state of every root token under the
original context (x, y_<i) and under the hindsight context (x, h, y_<i) of
Eq. (hindsight-contexts), the LM-head matrix W shared by both contexts, the
mask of tokens the policy generated itself (agent trajectories interleave environment
observations, Section 4.1 "Tasks"), and the continuation layout of Section 3.3
(each continuation reuses its root's prefix and, in this stand-in, has the
root's length and validity pattern).

Recipe, per workload, in this fixed draw order (index draws on a CPU
torch.Generator seeded with ``seed``; the large normal draws on a generator of
the target device seeded with ``seed + 1``):
  1. root lengths T_r ~ U{t_lo..t_hi};
  2. W ~ N(0, 0.02^2), fp32 [V, d];
  3. targets y_t ~ U{0..V-1};
  4. h_t = 3 * W[y_t] / ||W[y_t]||_2 + N(0, 1)^d  (original context);
  5. the validity mask (contiguous observation spans between action spans);
  6. the strongly perturbed positions (uniform / clustered spans / among valid);
  7. hindsight states = h + N(0, 0.05^2) everywhere, + N(0, 1) at perturbed rows;
  8. round-to-nearest-even cast to bf16 (fp32 workloads stay fp32).
Torch's generators are used because numpy's are ~20x too slow for the
10^9-element draws of the large workloads; values therefore depend on the
device they were drawn on, and every consumer uses the very tensors returned.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field
from typing import Optional

import torch

__all__ = ["Spec", "Workload", "SPECS", "sweep_spec", "small_spec", "generate"]


@dataclass(frozen=True)
class Spec:
    name: str
    n_roots: int
    t_lo: int                 # inclusive bounds of the root length T_r
    t_hi: int
    d: int                    # hidden size
    vocab: int                # V
    dtype: str                # "bf16" or "f32": hidden states and W
    k: int                    # branch points per root
    pert_frac: float          # fraction of strongly perturbed positions per root
    pert_mode: str = "uniform"  # "uniform" | "spans" | "valid"
    n_spans: int = 3          # for pert_mode == "spans"
    span_len: int = 32
    invalid_frac: float = 0.0   # fraction of tokens that are not policy-generated
    conts_per_root: Optional[int] = None   # continuations per root (default k)
    seed: int = 0

    @property
    def n_conts(self) -> int:
        return self.k if self.conts_per_root is None else self.conts_per_root


# The five workloads: tiny reference, math-, code- and agent-shaped rollouts.
SPECS = {
    "tiny": Spec("tiny", 4, 512, 512, 256, 4096, "f32", 4, 0.05),
    "math": Spec("math", 16, 256, 2048, 2048, 32000, "bf16", 8, 0.05,
                 conts_per_root=8),
    "code": Spec("code", 64, 512, 4096, 3584, 152064, "bf16", 8, 0.02,
                 pert_mode="spans"),
    "agent": Spec("agent", 32, 4096, 16384, 5120, 152064, "bf16", 16, 0.01,
                  pert_mode="valid", invalid_frac=0.20),
}

SWEEP_VOCABS = (32000, 128256, 256000)
SWEEP_TOKENS = (8192, 32768, 131072, 262144)


def sweep_spec(vocab: int, n_tokens: int, seed: int = 0) -> Spec:
    """Roofline sweep point: d = 4096, roots of 2048 tokens, k = 8."""
    assert n_tokens % 2048 == 0
    return Spec(f"sweep_V{vocab}_N{n_tokens}", n_tokens // 2048, 2048, 2048,
                4096, vocab, "bf16", 8, 0.05, seed=seed)


def small_spec(name: str = "small", **kw) -> Spec:
    """A reduced shape for fast tests; any field of Spec can be overridden."""
    base = dict(name=name, n_roots=3, t_lo=40, t_hi=300, d=128, vocab=1000,
                dtype="bf16", k=4, pert_frac=0.05)
    base.update(kw)
    return Spec(**base)


@dataclass
class Workload:
    spec: Spec
    h_orig: torch.Tensor        # [N, d] bf16/f32
    h_hind: torch.Tensor        # [N, d]
    w: torch.Tensor             # [V, d]
    targets: torch.Tensor       # [N] int32
    valid: torch.Tensor         # [N] uint8, 1 = policy-generated
    root_offsets: torch.Tensor  # [R + 1] int64
    perturbed: torch.Tensor     # [N] bool (information only)
    conts_per_root: torch.Tensor  # [R] int32
    cont_root: torch.Tensor     # [C] int32
    cont_offsets: torch.Tensor  # [C + 1] int64
    cont_valid: torch.Tensor    # [sum L_c] uint8
    lengths: list = field(default_factory=list)

    @property
    def n_tokens(self) -> int:
        return int(self.h_orig.shape[0])

    @property
    def n_roots(self) -> int:
        return self.spec.n_roots

    def to(self, device) -> "Workload":
        kw = {}
        for f in dataclasses.fields(self):
            v = getattr(self, f.name)
            kw[f.name] = v.to(device) if isinstance(v, torch.Tensor) else v
        return Workload(**kw)


def _rand_parts(total: int, parts: int, g: torch.Generator) -> list:
    """Split ``total`` into ``parts`` positive integers at random cut points."""
    if parts <= 1:
        return [total]
    cuts = torch.randperm(total - 1, generator=g)[: parts - 1] + 1
    cuts = sorted(cuts.tolist())
    bounds = [0] + cuts + [total]
    return [bounds[i + 1] - bounds[i] for i in range(parts)]


def _valid_pattern(T: int, frac: float, g: torch.Generator) -> torch.Tensor:
    """Contiguous observation spans (invalid) between action spans (valid)."""
    v = torch.ones(T, dtype=torch.uint8)
    n_inv = int(round(frac * T))
    if n_inv == 0:
        return v
    n_obs = int(torch.randint(4, 31, (1,), generator=g))   # <= 30 turns
    n_obs = max(1, min(n_obs, n_inv, (T - n_inv) - 1))
    obs = _rand_parts(n_inv, n_obs, g)
    act = _rand_parts(T - n_inv, n_obs + 1, g)
    pos = 0
    for i in range(n_obs):
        pos += act[i]
        v[pos:pos + obs[i]] = 0
        pos += obs[i]
    return v


def _perturbed_positions(spec: Spec, T: int, valid_r: torch.Tensor,
                         g: torch.Generator) -> torch.Tensor:
    n = int(round(spec.pert_frac * T))
    if spec.pert_mode == "uniform":
        pool = torch.arange(T)
    elif spec.pert_mode == "spans":
        L = min(spec.span_len, T)
        starts = torch.randint(0, T - L + 1, (spec.n_spans,), generator=g)
        pool = torch.unique(torch.cat([torch.arange(int(s), int(s) + L)
                                       for s in starts]))
    elif spec.pert_mode == "valid":
        pool = torch.nonzero(valid_r, as_tuple=False).flatten()
        n = int(round(spec.pert_frac * pool.numel()))
    else:
        raise ValueError(spec.pert_mode)
    n = min(n, pool.numel())
    return pool[torch.randperm(pool.numel(), generator=g)[:n]]


def generate(spec: Spec, device="cpu") -> Workload:
    """Draw one workload; every tensor is placed on ``device``."""
    device = torch.device(device)
    gc = torch.Generator().manual_seed(spec.seed)
    gd = torch.Generator(device=device).manual_seed(spec.seed + 1)
    R, d, V = spec.n_roots, spec.d, spec.vocab

    # 1. root lengths
    lengths = torch.randint(spec.t_lo, spec.t_hi + 1, (R,), generator=gc).tolist()
    N = sum(lengths)
    offs = [0]
    for T in lengths:
        offs.append(offs[-1] + T)

    # 2. LM head, fp32
    w = torch.randn(V, d, generator=gd, device=device) * 0.02
    # 3. targets
    targets = torch.randint(0, V, (N,), generator=gc, dtype=torch.int64)
    # 4. original-context states, peaked on the target row of W
    tgt_dev = targets.to(device)
    wy = w.index_select(0, tgt_dev)
    h = wy.mul_(3.0 / wy.norm(dim=1, keepdim=True))
    del wy
    h.add_(torch.randn(N, d, generator=gd, device=device))

    # 5. validity mask
    valid = torch.ones(N, dtype=torch.uint8)
    if spec.invalid_frac > 0:
        for r, T in enumerate(lengths):
            valid[offs[r]:offs[r + 1]] = _valid_pattern(T, spec.invalid_frac, gc)
    # 6. strongly perturbed positions
    perturbed = torch.zeros(N, dtype=torch.bool)
    for r, T in enumerate(lengths):
        p = _perturbed_positions(spec, T, valid[offs[r]:offs[r + 1]], gc)
        perturbed[offs[r] + p] = True

    # 7. hindsight states
    hh = h + torch.randn(N, d, generator=gd, device=device) * 0.05
    rows = torch.nonzero(perturbed, as_tuple=False).flatten().to(device)
    if rows.numel():
        hh.index_add_(0, rows, torch.randn(rows.numel(), d, generator=gd,
                                           device=device))

    # 8. cast
    if spec.dtype == "bf16":
        w, h, hh = w.to(torch.bfloat16), h.to(torch.bfloat16), hh.to(torch.bfloat16)
    elif spec.dtype != "f32":
        raise ValueError(spec.dtype)

    # continuation layout: C_r continuations per root, each of the root's
    # length and validity pattern (the sampled suffix is not modelled)
    C = spec.n_conts
    cont_root, cont_len, cont_valid = [], [], []
    for r, T in enumerate(lengths):
        for _ in range(C):
            cont_root.append(r)
            cont_len.append(T)
            cont_valid.append(valid[offs[r]:offs[r + 1]])
    coffs = [0]
    for L in cont_len:
        coffs.append(coffs[-1] + L)
    cv = torch.cat(cont_valid) if cont_valid else torch.zeros(0, dtype=torch.uint8)

    i64 = dict(dtype=torch.int64, device=device)
    return Workload(
        spec=spec,
        h_orig=h.contiguous(), h_hind=hh.contiguous(), w=w.contiguous(),
        targets=targets.to(device=device, dtype=torch.int32),
        valid=valid.to(device),
        root_offsets=torch.tensor(offs, **i64),
        perturbed=perturbed.to(device),
        conts_per_root=torch.full((R,), C, dtype=torch.int32, device=device),
        cont_root=torch.tensor(cont_root, dtype=torch.int32, device=device),
        cont_offsets=torch.tensor(coffs, **i64),
        cont_valid=cv.to(device),
        lengths=lengths,
    )
