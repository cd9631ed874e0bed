"""The HBM-bound kernels at the sizes their bandwidth is measured on
(`bench.py --micro`): selection over 8192 roots x 4096 tokens, suffix masks
over 32768 continuations x 4096 tokens, the GRPO update over 16384
trajectories x 4096 tokens -- every output against the oracle (selection and
masks bit for bit)."""
import numpy as np
import pytest
import torch

import oracle
from tests.helpers import check_grpo

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hdl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as m
    return m


def test_select_scaled(hdl):
    R, T, k = 8192, 4096, 8
    g = torch.Generator(device="cuda").manual_seed(0)
    delta = torch.rand(R * T, generator=g, device="cuda")
    valid = (torch.rand(R * T, generator=g, device="cuda") < 0.8).to(torch.uint8)
    offs = torch.arange(0, R * T + 1, T, dtype=torch.int64, device="cuda")
    bp, ns, bd = hdl.hdl_select_branches(delta, valid, offs, k)
    pos, nsel, val = oracle.select_branches(delta.cpu().numpy().astype(np.float64),
                                            valid.cpu().numpy(), offs.cpu().numpy(), k)
    assert np.array_equal(ns.cpu().numpy(), nsel)
    assert np.array_equal(bp.cpu().numpy(), pos)
    assert np.array_equal(bd.cpu().numpy().astype(np.float64), val, equal_nan=True)


def test_mask_scaled(hdl):
    C, L = 32768, 4096
    g = torch.Generator(device="cuda").manual_seed(1)
    offs = torch.arange(0, C * L + 1, L, dtype=torch.int64, device="cuda")
    cb = torch.randint(-1, L, (C,), generator=g, device="cuda", dtype=torch.int32)
    valid = (torch.rand(C * L, generator=g, device="cuda") < 0.8).to(torch.uint8)
    m = hdl.hdl_suffix_mask(cb, offs, valid)
    ref = oracle.suffix_mask(cb.cpu().numpy(), offs.cpu().numpy(), valid.cpu().numpy())
    assert np.array_equal(m.cpu().numpy(), ref)


def test_grpo_scaled(hdl):
    J, L, G = 16384, 4096, 16
    T = J * L
    g = torch.Generator(device="cuda").manual_seed(2)
    lpo = -torch.rand(T, generator=g, device="cuda") * 3
    lpn = lpo + torch.randn(T, generator=g, device="cuda") * 0.3
    m = (torch.rand(T, generator=g, device="cuda") < 0.7).to(torch.uint8)
    toffs = torch.arange(0, T + 1, L, dtype=torch.int64, device="cuda")
    R = torch.rand(J, generator=g, device="cuda")
    goffs = torch.arange(0, J + 1, G, dtype=torch.int32, device="cuda")
    adv, grad, stats = hdl.hdl_grpo_loss(lpn, lpo, m, toffs, R, goffs)
    check_grpo(adv.cpu().numpy(), grad.cpu().numpy(), stats.cpu().numpy(), lpn.cpu().numpy(),
               lpo.cpu().numpy(), m.cpu().numpy(), toffs.cpu().numpy(), R.cpu().numpy(),
               goffs.cpu().numpy())
