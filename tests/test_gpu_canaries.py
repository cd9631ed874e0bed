"""Out-of-bounds write checks without compute-sanitizer: every output buffer
of every entry point is placed between guard bands filled with a byte
pattern, the calls run on ragged shapes, and the guard bytes must be intact
afterwards (and the outputs must still be the ones the unguarded call
gives)."""
import numpy as np
import pytest
import torch

import hdl_synth

pytestmark = pytest.mark.gpu

GUARD = 4096          # bytes on each side
PATTERN = 0xA5


@pytest.fixture(scope="module")
def hdl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as m
    return m


class Guarded:
    """A device tensor of `shape`/`dtype` inside a byte buffer with guards."""

    def __init__(self, shape, dtype, align=256, offset=0):
        n = int(np.prod(shape)) if len(shape) else 1
        nbytes = n * torch.empty(0, dtype=dtype).element_size()
        self.raw = torch.full((GUARD + nbytes + GUARD + align,), PATTERN, dtype=torch.uint8,
                              device="cuda")
        base = self.raw.data_ptr()
        pad = (-(base + GUARD)) % align
        self.lo = GUARD + pad + offset
        self.hi = self.lo + nbytes
        self.t = self.raw[self.lo:self.hi].view(dtype).view(shape)

    def intact(self):
        r = self.raw.cpu().numpy()
        return bool(np.all(r[:self.lo] == PATTERN) and np.all(r[self.hi:] == PATTERN))


SHAPES = [(1, 64, 1), (129, 128, 257), (300, 256, 4097), (700, 192, 9000)]


@pytest.mark.parametrize("n,d,V", SHAPES)
def test_rescore_writes_stay_in_bounds(hdl, n, d, V):
    spec = hdl_synth.small_spec("g", n_roots=1, t_lo=n, t_hi=n, d=d, vocab=V, seed=n)
    wl = hdl_synth.generate(spec, device="cuda")
    ref = hdl.hdl_rescore_ex(wl.h_orig, wl.h_hind, wl.w, wl.targets, want_entropy_hind=True)
    outs = [Guarded((n,), torch.float32) for _ in range(5)]
    need = hdl.hdl_rescore_ex_workspace_bytes(n, d, V, entropy=True)
    ws = Guarded((need,), torch.uint8)
    hdl.hdl_rescore_ex(wl.h_orig, wl.h_hind, wl.w, wl.targets, outs[0].t, outs[1].t, outs[2].t,
                       outs[3].t, outs[4].t, workspace=ws.t)
    torch.cuda.synchronize()
    for g in outs + [ws]:
        assert g.intact()
    for g, r in zip(outs, (ref[0], ref[1], ref[2], ref[3], ref[4])):
        assert torch.equal(g.t, r)
    # shard statistics
    st = Guarded((2, n, 4), torch.float32)
    sws = Guarded((hdl.hdl_rescore_shard_workspace_bytes(n, d, V),), torch.uint8)
    hdl.hdl_rescore_shard(wl.h_orig, wl.h_hind, wl.w, wl.targets, 0, stats=st.t, workspace=sws.t)
    torch.cuda.synchronize()
    assert st.intact() and sws.intact()


def test_select_assign_mask_stay_in_bounds(hdl):
    rng = np.random.default_rng(3)
    lengths = list(rng.integers(0, 600, size=400)) + [9000, 0, 3]
    R, k = len(lengths), 7
    offs = torch.tensor(np.concatenate([[0], np.cumsum(lengths)]), dtype=torch.int64,
                        device="cuda")
    N = int(offs[-1])
    delta = torch.rand(N, device="cuda")
    valid = (torch.rand(N, device="cuda") < 0.8).to(torch.uint8)
    for R_used in (R, 5):                         # warp-per-root and 16-warp paths
        o = offs[:R_used + 1]
        bp, ns, bd = Guarded((R_used, k), torch.int32), Guarded((R_used,), torch.int32), \
            Guarded((R_used, k), torch.float32)
        hdl.hdl_select_branches(delta, valid, o, k, branch_pos=bp.t, n_selected=ns.t,
                                branch_delta=bd.t)
        torch.cuda.synchronize()
        assert bp.intact() and ns.intact() and bd.intact()
    conts = torch.randint(0, 9, (R,), dtype=torch.int32, device="cuda")
    C = int(conts.sum())
    cb = Guarded((C,), torch.int32)
    nsel = torch.randint(0, k + 1, (R,), dtype=torch.int32, device="cuda")
    pos = torch.randint(0, 500, (R, k), dtype=torch.int32, device="cuda")
    hdl.hdl_assign_continuations(nsel, pos, conts, cont_branch=cb.t)
    torch.cuda.synchronize()
    assert cb.intact()
    lens = rng.integers(0, 300, size=C)
    coffs = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int64, device="cuda")
    total = int(coffs[-1])
    cv_all = (torch.rand(total + 16, device="cuda") < 0.7).to(torch.uint8)
    # (mask, validity) offsets from 16-byte alignment: vector path, byte path,
    # phase-shifted vector path
    for offset, v_off in ((0, 0), (1, 0), (3, 3)):
        m = Guarded((total,), torch.uint8, offset=offset)
        cv = cv_all[v_off:v_off + total]
        hdl.hdl_suffix_mask(cb.t, coffs, cv, mask=m.t)
        torch.cuda.synchronize()
        assert m.intact()


@pytest.mark.parametrize("phase", [0, 1, 3])
def test_grpo_stays_in_bounds(hdl, phase):
    """Token streams `phase` elements off 16-byte alignment (all four alike:
    the vector path, shifted when phase > 0)."""
    rng = np.random.default_rng(4)
    sizes = rng.integers(1, 17, size=50)
    goffs = torch.tensor(np.concatenate([[0], np.cumsum(sizes)]), dtype=torch.int32,
                         device="cuda")
    J = int(goffs[-1])
    lens = rng.integers(0, 700, size=J)
    toffs = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int64,
                         device="cuda")
    T = int(toffs[-1])
    lpo = -torch.rand(T + phase, device="cuda")[phase:]
    lpn = (lpo + 0.3 * torch.randn(T, device="cuda"))
    lpn = torch.cat([torch.zeros(phase, device="cuda"), lpn])[phase:]
    m = (torch.rand(T + phase, device="cuda") < 0.7).to(torch.uint8)[phase:]
    R = torch.rand(J, device="cuda")
    adv, grad, st = Guarded((J,), torch.float32), \
        Guarded((T,), torch.float32, offset=4 * phase), Guarded((4,), torch.float32)
    ws = Guarded((hdl.hdl_grpo_loss_workspace_bytes(),), torch.uint8)
    hdl.hdl_grpo_loss(lpn, lpo, m, toffs, R, goffs, advantages=adv.t, grad=grad.t, stats=st.t,
                      workspace=ws.t)
    torch.cuda.synchronize()
    for g in (adv, grad, st, ws):
        assert g.intact()
