"""The GRPO update after branch selection on the GPU against the oracle:
group-relative advantages and the asymmetric-clip token-level loss and its
gradient on suffix-only masks (Sections 3, 3.3, 4.1)."""
import numpy as np
import pytest
import torch

from tests.helpers import check_grpo

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hdl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as m
    return m


def make_batch(seed, n_groups, max_len):
    rng = np.random.default_rng(seed)
    sizes = rng.integers(1, 17, size=n_groups)
    sizes[:2] = [16, 1]                               # a full group and a lone trajectory
    goffs = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int32)
    J = int(goffs[-1])
    lens = rng.integers(0, max_len, size=J)
    toffs = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    T = int(toffs[-1])
    rewards = rng.random(J).astype(np.float32)
    rewards[goffs[2]:goffs[3]] = 0.5                  # uniform rewards: zero advantage
    lpo = (-rng.exponential(size=T)).astype(np.float32)
    lpn = (lpo + rng.normal(scale=0.3, size=T)).astype(np.float32)   # ratios across the clip
    mask = (rng.random(T) < 0.7).astype(np.uint8)
    return lpn, lpo, mask, toffs, rewards, goffs


# (3, 20000, 21): ~170K short (and empty) trajectories, so that a warp's
# share of the tokens spans more than 31 of them
@pytest.mark.parametrize("seed,n_groups,max_len", [(0, 40, 300), (1, 8, 5000), (2, 300, 30),
                                                   (3, 20000, 21)])
def test_grpo_loss_matches_oracle(hdl, seed, n_groups, max_len):
    lpn, lpo, mask, toffs, R, goffs = make_batch(seed, n_groups, max_len)
    t = lambda x: torch.from_numpy(x).cuda()
    adv, grad, stats = hdl.hdl_grpo_loss(t(lpn), t(lpo), t(mask), t(toffs), t(R), t(goffs))
    check_grpo(adv.cpu().numpy(), grad.cpu().numpy(), stats.cpu().numpy(), lpn, lpo, mask,
               toffs, R, goffs)


def test_grpo_paper_group(hdl):
    """One problem of the paper's default layout: 2 roots + 2 x (3 + 4)
    continuations = G = 16 (Section 4.1); equal rewards give zero loss."""
    goffs = np.array([0, 16], np.int32)
    lens = np.full(16, 50)
    toffs = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    R = np.full(16, 1.0, np.float32)
    lp = np.full(800, -0.5, np.float32)
    mask = np.ones(800, np.uint8)
    t = lambda x: torch.from_numpy(x).cuda()
    adv, grad, stats = hdl.hdl_grpo_loss(t(lp), t(lp), t(mask), t(toffs), t(R), t(goffs))
    assert torch.all(adv == 0) and stats[0].item() == 0 and stats[1].item() == 800
    assert torch.all(grad == 0)


@pytest.mark.parametrize("shift", [1, 2, 3])
@pytest.mark.parametrize("grad_off", [None, 1, 2])
def test_grpo_unaligned(hdl, shift, grad_off):
    """First trajectory starting at a token that is not a multiple of 4, and
    buffers that are not 16-byte aligned: all four token streams one element
    off (the phase-shifted vector path: grad_off 1), the gradient at another
    offset (grad_off None: a fresh aligned buffer, or 2), which takes the
    scalar path."""
    lpn, lpo, mask, toffs, R, goffs = make_batch(10 + shift, 30, 200)
    # `shift` leading tokens outside every trajectory, carrying no loss
    pad = lambda x, v: np.concatenate([np.full(shift, v, x.dtype), x])
    lpn2, lpo2, mask2 = pad(lpn, -1.0), pad(lpo, -1.0), pad(mask, 0)
    toffs2 = toffs + shift
    buf = lambda x: torch.from_numpy(np.concatenate([x[:1], x])).cuda()[1:]   # misalign
    grad = None
    if grad_off is not None:
        grad = torch.full((len(lpn2) + grad_off,), 5.0, device="cuda")[grad_off:]
    adv, grad, stats = hdl.hdl_grpo_loss(buf(lpn2), buf(lpo2), buf(mask2),
                                         torch.from_numpy(toffs2).cuda(),
                                         torch.from_numpy(R).cuda(),
                                         torch.from_numpy(goffs).cuda(), grad=grad)
    g = grad.cpu().numpy()
    assert np.all(g[:shift] == 0)
    check_grpo(adv.cpu().numpy(), g, stats.cpu().numpy(), lpn, lpo, mask, toffs, R, goffs,
               grad_slice=slice(shift, None))


def test_grpo_empty_inputs(hdl):
    """No tokens and no trajectories: the call succeeds and every statistic is
    0.  Groups but no tokens: the advantages are still R - group mean."""
    e32 = torch.empty(0, dtype=torch.float32, device="cuda")
    eu8 = torch.empty(0, dtype=torch.uint8, device="cuda")
    zero64 = torch.zeros(1, dtype=torch.int64, device="cuda")
    zero32 = torch.zeros(1, dtype=torch.int32, device="cuda")
    adv, grad, stats = hdl.hdl_grpo_loss(e32, e32, eu8, zero64, e32, zero32)
    assert adv.numel() == 0 and torch.all(stats == 0)
    R = np.array([0.25, 1.0, 0.5], dtype=np.float32)
    adv, grad, stats = hdl.hdl_grpo_loss(
        e32, e32, eu8, torch.zeros(4, dtype=torch.int64, device="cuda"),
        torch.from_numpy(R).cuda(), torch.tensor([0, 3], dtype=torch.int32, device="cuda"))
    assert np.allclose(adv.cpu().numpy(), R - R.astype(np.float64).mean(), rtol=0, atol=1e-7)
    assert torch.all(stats == 0)
