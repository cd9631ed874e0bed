"""Selection, allocation and mask kernels: bit-exact against the oracle when
fed the same scores, offsets and masks (Sections 3.2, 3.3, 4.1, 4.4)."""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hdl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as m
    return m


def make_roots(lengths, seed, tie_levels=None, nan_frac=0.0, invalid_frac=0.2):
    rng = np.random.default_rng(seed)
    offs = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    N = int(offs[-1])
    if tie_levels:
        delta = (rng.integers(0, tie_levels, size=N) * 0.25).astype(np.float32)
    else:
        delta = rng.exponential(size=N).astype(np.float32)
    if nan_frac:
        delta[rng.random(N) < nan_frac] = np.nan
    valid = (rng.random(N) >= invalid_frac).astype(np.uint8)
    return delta, valid, offs


def shifted(x: np.ndarray, off: int) -> torch.Tensor:
    """x on the GPU starting `off` elements into a fresh (aligned) buffer."""
    buf = torch.zeros(len(x) + off, dtype=torch.from_numpy(x[:0]).dtype, device="cuda")
    buf[off:] = torch.from_numpy(x).cuda()
    return buf[off:]


# element offsets of (scores, validity): the same residue mod 4 keeps the
# 16-byte path (shifted to the common phase), different ones take the
# element-by-element path
OFFSETS = [(1, 1), (3, 3), (1, 2), (2, 0)]


def gpu_select(hdl, delta, valid, offs, k, **kw):
    d = torch.from_numpy(delta).cuda()
    v = None if valid is None else torch.from_numpy(valid).cuda()
    o = torch.from_numpy(offs).cuda()
    bp, ns, bd = hdl.hdl_select_branches(d, v, o, k, **kw)
    return bp.cpu().numpy(), ns.cpu().numpy(), bd.cpu().numpy()


def assert_select_equal(hdl, delta, valid, offs, k, **kw):
    bp, ns, bd = gpu_select(hdl, delta, valid, offs, k, **kw)
    pos, nsel, val = oracle.select_branches(delta.astype(np.float64), valid, offs, k, **kw)
    assert np.array_equal(ns, nsel)
    assert np.array_equal(bp, pos)
    assert np.array_equal(bd.astype(np.float64), val, equal_nan=True)


CASES = [
    (list(np.random.default_rng(5).integers(0, 300, size=700)), 8, {}),   # warp per root
    (list(np.random.default_rng(6).integers(0, 70, size=400)), 16, {}),
    (list(np.random.default_rng(7).integers(0, 900, size=350)), 3, {}),
    (list(np.random.default_rng(8).integers(1024, 3000, size=330)), 8, {}),   # 4 warps / root
    (list(np.random.default_rng(9).integers(8192, 8800, size=310)), 5, {}),   # 16 warps / root
    ([0, 1, 2, 3, 17, 100, 511, 513, 4096], 4, {}),
    ([16384, 16384, 12000], 16, {}),                       # maximum k, long roots
    ([3, 5, 1, 0, 2], 8, {}),                              # k > T
    ([1000] * 40, 8, {}),                                  # many roots
]


@pytest.mark.parametrize("lengths,k,kw", CASES)
def test_select_plain(hdl, lengths, k, kw):
    for seed, ties in ((0, None), (1, 3), (2, 1)):        # distinct, heavy ties, all equal
        delta, valid, offs = make_roots(lengths, seed, tie_levels=ties)
        assert_select_equal(hdl, delta, valid, offs, k, **kw)
        assert_select_equal(hdl, delta, None, offs, k, **kw)


def test_select_nan_negative_zero_and_all_invalid(hdl):
    delta, valid, offs = make_roots([200, 50, 300], 5, nan_frac=0.3)
    delta[:10] = -0.0
    delta[10:20] = 0.0
    delta[20:25] = -1.5
    delta[25] = np.inf
    valid[offs[1]:offs[2]] = 0                            # a root with no candidate
    for k in (0, 1, 5, 16):
        assert_select_equal(hdl, delta, valid, offs, k)


def test_select_window(hdl):
    delta, valid, offs = make_roots([500, 20, 1000], 6)
    for lo, hi in ((0, 0), (10, 0), (0, 100), (50, 60), (600, 0), (5, 3)):
        assert_select_equal(hdl, delta, valid, offs, 8, lo=lo, hi=hi)


def add_spikes(delta, offs, seed, spans=3, width=32, lift=5.0):
    """Clustered high scores (the shape divergence takes around a decisive
    token): `spans` runs of `width` positions per root lifted by `lift`."""
    rng = np.random.default_rng(seed)
    for r in range(len(offs) - 1):
        T = int(offs[r + 1] - offs[r])
        for _ in range(spans if T > width else 0):
            a = int(offs[r]) + int(rng.integers(0, T - width))
            delta[a:a + width] += lift
    return delta


@pytest.mark.parametrize("gap_mode", [0, 1])
def test_select_spacing_many_roots(hdl, gap_mode):
    """The spacing rule with many roots (one warp per root; greedy keeps a
    per-thread list and rescans only when it runs dry), clustered scores so
    that whole runs are ruled out at once, gaps from 1 (plain top-k) to longer
    than the roots, windows, ties, NaN and +-inf: bit-exact against the
    oracle."""
    rng = np.random.default_rng(40 + gap_mode)
    lengths = list(rng.integers(0, 2000, size=400)) + [0, 1, 2, 3, 4, 5, 40, 70000]
    for seed, ties in ((0, None), (1, 4)):
        delta, valid, offs = make_roots(lengths, 50 + seed, tie_levels=ties, nan_frac=0.01)
        delta = add_spikes(delta, offs, seed)
        delta[::997] = np.inf
        delta[5::1013] = -np.inf
        for k in (1, 8, 16):
            for min_gap in (1, 3, 40, 5000):
                assert_select_equal(hdl, delta, valid, offs, k, min_gap=min_gap,
                                    gap_mode=gap_mode)
        for lo, hi in ((10, 0), (100, 900)):
            assert_select_equal(hdl, delta, None, offs, 8, min_gap=20, gap_mode=gap_mode,
                                lo=lo, hi=hi)


@pytest.mark.parametrize("d_off,v_off", [(1, 1), (1, 2)])
@pytest.mark.parametrize("n_roots", [7, 500])
@pytest.mark.parametrize("gap_mode", [0, 1])
def test_select_spacing_unaligned(hdl, n_roots, gap_mode, d_off, v_off):
    """Scores / validity off their 16- / 4-byte alignment: both spacing modes
    on the phase-shifted vector path and on the scalar path, with few and
    with many roots."""
    lengths = list(np.random.default_rng(n_roots).integers(0, 2500, size=n_roots))
    delta, valid, offs = make_roots(lengths, 13, tie_levels=6)
    delta = add_spikes(delta, offs, 3)
    d, v = shifted(delta, d_off), shifted(valid, v_off)
    o = torch.from_numpy(offs).cuda()
    for min_gap in (2, 33):
        bp, ns, bd = hdl.hdl_select_branches(d, v, o, 16, min_gap=min_gap, gap_mode=gap_mode)
        pos, nsel, val = oracle.select_branches(delta.astype(np.float64), valid, offs, 16,
                                                min_gap=min_gap, gap_mode=gap_mode)
        assert np.array_equal(ns.cpu().numpy(), nsel)
        assert np.array_equal(bp.cpu().numpy(), pos)
        assert np.array_equal(bd.cpu().numpy().astype(np.float64), val, equal_nan=True)


@pytest.mark.parametrize("gap_mode", [0, 1])
@pytest.mark.parametrize("min_gap", [1, 2, 7, 64])
def test_select_spacing(hdl, gap_mode, min_gap):
    for seed, ties in ((7, None), (8, 3)):
        delta, valid, offs = make_roots([0, 5, 40, 300, 2048, 9000], seed, tie_levels=ties)
        # cluster the large scores so that the spacing rule bites
        delta[offs[4] + 100:offs[4] + 140] += 5
        assert_select_equal(hdl, delta, valid, offs, 8, min_gap=min_gap, gap_mode=gap_mode)
        assert_select_equal(hdl, delta, valid, offs, 16, min_gap=min_gap, gap_mode=gap_mode)


def test_select_nonmonotone_offsets_are_empty(hdl):
    delta, valid, offs = make_roots([100, 100], 9)
    offs = np.array([0, 100, 50], dtype=np.int64)         # second root ends before it starts
    bp, ns, bd = gpu_select(hdl, delta, valid, offs, 4)
    assert ns[1] == 0 and np.all(bp[1] == -1)


@pytest.mark.parametrize("extra_to_higher", [True, False])
def test_assign_continuations(hdl, extra_to_higher):
    rng = np.random.default_rng(11)
    R, k = 300, 8
    nsel = rng.integers(0, k + 1, size=R).astype(np.int32)
    pos = np.full((R, k), -1, np.int32)
    for r in range(R):
        pos[r, :nsel[r]] = rng.choice(5000, size=nsel[r], replace=False)
    conts = rng.integers(0, 20, size=R).astype(np.int32)
    conts[:3] = [7, 7, 3]
    ref = oracle.assign_continuations(nsel, pos, conts, extra_to_higher)
    cb = hdl.hdl_assign_continuations(torch.from_numpy(nsel).cuda(), torch.from_numpy(pos).cuda(),
                                      torch.from_numpy(conts).cuda(), extra_to_higher,
                                      n_cont=int(conts.sum()))
    assert np.array_equal(cb.cpu().numpy(), ref)


def test_assign_paper_configs(hdl):
    """2x2 -> 3+4, 2x1 -> 7, 4x2 -> 1+2 per root (Section 4.1, Table fork-ablation)."""
    for roots, pts, C, counts in ((2, 2, 7, [4, 3]), (2, 1, 7, [7]), (4, 2, 3, [2, 1])):
        nsel = torch.full((roots,), pts, dtype=torch.int32, device="cuda")
        pos = torch.arange(roots * pts, dtype=torch.int32, device="cuda").view(roots, pts) * 10
        conts = torch.full((roots,), C, dtype=torch.int32, device="cuda")
        cb = hdl.hdl_assign_continuations(nsel, pos, conts, n_cont=roots * C).cpu().numpy()
        for r in range(roots):
            seg = cb[r * C:(r + 1) * C]
            got = [int((seg == p).sum()) for p in pos[r].cpu().numpy()]
            assert got == counts


def test_assign_capacity_is_respected(hdl):
    nsel = torch.tensor([2, 2], dtype=torch.int32, device="cuda")
    pos = torch.tensor([[1, 2], [3, 4]], dtype=torch.int32, device="cuda")
    conts = torch.tensor([7, 7], dtype=torch.int32, device="cuda")
    out = torch.full((20,), -7, dtype=torch.int32, device="cuda")
    hdl.hdl_assign_continuations(nsel, pos, conts, cont_branch=out[:10])
    o = out.cpu().numpy()
    assert np.array_equal(o[:10], [1, 1, 1, 1, 2, 2, 2, 3, 3, 3]) and np.all(o[10:] == -7)


def mask_case(seed, n_cont, max_len):
    rng = np.random.default_rng(seed)
    lens = rng.integers(0, max_len, size=n_cont)
    lens[:4] = [0, 1, 15, 17]
    offs = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    br = np.array([rng.integers(-1, L + 3) if L > 0 else rng.integers(-1, 3) for L in lens],
                  dtype=np.int32)
    valid = (rng.random(int(offs[-1])) < 0.8).astype(np.uint8)
    return br, offs, valid


@pytest.mark.parametrize("seed,n_cont,max_len", [(0, 50, 300), (1, 600, 40), (2, 9, 20000)])
def test_suffix_mask(hdl, seed, n_cont, max_len):
    br, offs, valid = mask_case(seed, n_cont, max_len)
    ref = oracle.suffix_mask(br, offs, valid)
    ref_nv = oracle.suffix_mask(br, offs, None)
    tb, to, tv = (torch.from_numpy(x).cuda() for x in (br, offs, valid))
    m = hdl.hdl_suffix_mask(tb, to, tv)
    assert np.array_equal(m.cpu().numpy(), ref)
    m = hdl.hdl_suffix_mask(tb, to, None, mask_len=int(offs[-1]))
    assert np.array_equal(m.cpu().numpy(), ref_nv)


def test_suffix_mask_unaligned_and_offset_range(hdl):
    """Mask and validity bytes at the same offset from 16-byte alignment (the
    phase-shifted vector path), at different ones (the byte path), and a
    range that starts and ends mid-buffer: bytes outside the continuations
    stay untouched."""
    br, offs, valid = mask_case(3, 40, 200)
    total = int(offs[-1])
    shift = 5
    L = total + 2 * shift
    ref = oracle.suffix_mask(br, offs, valid)
    o = torch.from_numpy(offs + shift).cuda()
    for mbase, vbase in ((0, 0), (1, 1), (7, 7), (1, 3), (0, 9)):
        mbuf = torch.full((L + mbase,), 7, dtype=torch.uint8, device="cuda")
        vbuf = torch.zeros(L + vbase, dtype=torch.uint8, device="cuda")
        vbuf[vbase + shift:vbase + shift + total] = torch.from_numpy(valid).cuda()
        hdl.hdl_suffix_mask(torch.from_numpy(br).cuda(), o, vbuf[vbase:], mask=mbuf[mbase:])
        got = mbuf[mbase:].cpu().numpy()
        assert np.all(got[:shift] == 7) and np.all(got[shift + total:] == 7)
        assert np.array_equal(got[shift:shift + total], ref)


@pytest.mark.parametrize("d_off,v_off", OFFSETS)
@pytest.mark.parametrize("n_roots", [5, 600])
def test_select_unaligned_buffers(hdl, n_roots, d_off, v_off):
    """Scores / validity off their 16- / 4-byte alignment: the phase-shifted
    vector path when both are off by the same amount, else the scalar path."""
    lengths = list(np.random.default_rng(n_roots).integers(0, 500, size=n_roots))
    delta, valid, offs = make_roots(lengths, 12, tie_levels=5)
    bp, ns, bd = hdl.hdl_select_branches(shifted(delta, d_off), shifted(valid, v_off),
                                         torch.from_numpy(offs).cuda(), 8)
    pos, nsel, val = oracle.select_branches(delta.astype(np.float64), valid, offs, 8)
    assert np.array_equal(ns.cpu().numpy(), nsel) and np.array_equal(bp.cpu().numpy(), pos)
    assert np.array_equal(bd.cpu().numpy().astype(np.float64), val, equal_nan=True)


_SPLIT_SCRIPT = r"""
import sys
import numpy as np
import torch
sys.path.insert(0, sys.argv[1])
import paper_2609_36864_gb300 as hdl
data = np.load(sys.argv[2])
d = torch.from_numpy(data["delta"]).cuda()
v = torch.from_numpy(data["valid"]).cuda()
o = torch.from_numpy(data["offs"]).cuda()
out = {}
for k in (1, 8, 16):
    for lo, hi in ((0, 0), (37, 3001)):
        bp, ns, bd = hdl.hdl_select_branches(d, v, o, k, lo=lo, hi=hi)
        out[f"bp{k}_{lo}"] = bp.cpu().numpy()
        out[f"ns{k}_{lo}"] = ns.cpu().numpy()
        out[f"bd{k}_{lo}"] = bd.cpu().numpy()
    bp, ns, bd = hdl.hdl_select_branches(d, v, o, k, min_gap=6, gap_mode=1)
    out[f"bp{k}_drop"], out[f"ns{k}_drop"] = bp.cpu().numpy(), ns.cpu().numpy()
np.savez(sys.argv[3], **out)
"""


@pytest.mark.parametrize("split", ["1", "2", "4", "8"])
def test_select_warps_per_root(hdl, tmp_path, split):
    """The many-roots mode with 1, 2, 4 or 8 warps per root (forced): every
    split gives the oracle's selection bit for bit, including ragged and
    empty roots, heavy ties and a window."""
    rng = np.random.default_rng(21)
    lengths = list(rng.integers(1500, 6000, size=330)) + [0, 1, 5, 4099]
    delta, valid, offs = make_roots(lengths, 22, tie_levels=40)
    inp = tmp_path / "in.npz"
    np.savez(inp, delta=delta, valid=valid, offs=offs)
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    outp = tmp_path / "out.npz"
    subprocess.run([sys.executable, "-c", _SPLIT_SCRIPT, root, str(inp), str(outp)],
                   env=dict(os.environ, HDL_SELECT_SPLIT=split), check=True, timeout=300)
    got = np.load(outp)
    for k in (1, 8, 16):
        for lo, hi in ((0, 0), (37, 3001)):
            pos, nsel, val = oracle.select_branches(delta.astype(np.float64), valid, offs, k,
                                                    lo=lo, hi=hi)
            assert np.array_equal(got[f"ns{k}_{lo}"], nsel)
            assert np.array_equal(got[f"bp{k}_{lo}"], pos)
            assert np.array_equal(got[f"bd{k}_{lo}"].astype(np.float64), val, equal_nan=True)
        pos, nsel, _ = oracle.select_branches(delta.astype(np.float64), valid, offs, k,
                                              min_gap=6, gap_mode=1)
        assert np.array_equal(got[f"ns{k}_drop"], nsel)
        assert np.array_equal(got[f"bp{k}_drop"], pos)


def test_select_randomized(hdl):
    """40 seeded random configurations around the launch-mode boundaries
    (2 roots per SM; few long roots, where the heuristic splits a root over
    several warps; many short ones), with windows, ties, NaNs, invalid runs
    and every k: bit-exact against the oracle."""
    rng = np.random.default_rng(2024)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    for case in range(40):
        kind = case % 4
        if kind == 0:
            R = int(rng.integers(2 * sms - 3, 2 * sms + 4))
            lengths = rng.integers(0, 3000, size=R)
        elif kind == 1:
            R = int(rng.integers(2 * sms, 2 * sms + 200))
            lengths = rng.integers(8000, 20000, size=R)
        elif kind == 2:
            R = int(rng.integers(1, 40))
            lengths = rng.integers(0, 20000, size=R)
        else:
            R = int(rng.integers(1000, 3000))
            lengths = rng.integers(0, 400, size=R)
        ties = [None, 2, 50][case % 3]
        delta, valid, offs = make_roots(list(lengths), 100 + case, tie_levels=ties,
                                        nan_frac=0.01 * (case % 2),
                                        invalid_frac=float(rng.choice([0.0, 0.2, 0.9])))
        k = int(rng.integers(1, 17))
        lo, hi = [(0, 0), (int(rng.integers(0, 500)), 0), (0, int(rng.integers(1, 9000))),
                  (int(rng.integers(0, 300)), int(rng.integers(300, 12000)))][case % 4]
        assert_select_equal(hdl, delta, valid if case % 5 else None, offs, k, lo=lo, hi=hi)


def runs_case(seed, n_roots=1700):
    """Many roots (more than the resident warps): mostly short, some empty,
    and every 97th one long (3000-12000 positions)."""
    rng = np.random.default_rng(seed)
    lengths = rng.integers(0, 120, size=n_roots)
    lengths[::13] = 0
    lengths[5::97] = rng.integers(3000, 12000, size=len(lengths[5::97]))
    return make_roots(list(lengths), seed + 1, tie_levels=30, nan_frac=0.01)


@pytest.mark.parametrize("d_off,v_off", OFFSETS)
def test_select_many_roots_unaligned_and_nonmonotone(hdl, d_off, v_off):
    """1700 ragged roots (short, empty and long ones) on buffers off their
    alignment (the phase-shifted vector path and the element-by-element one),
    with a few roots whose end precedes their start: the oracle's result bit
    for bit."""
    delta, valid, offs = runs_case(40 + d_off + 4 * v_off)
    offs = offs.copy()
    for r in (7, 600, 1333):                      # end before start: an empty root
        offs[r + 1] = offs[r] - 3 if offs[r] >= 3 else offs[r + 1]
    for k in (4, 16):
        bp, ns, bd = hdl.hdl_select_branches(shifted(delta, d_off), shifted(valid, v_off),
                                             torch.from_numpy(offs).cuda(), k)
        pos, nsel, val = oracle.select_branches(delta.astype(np.float64), valid, offs, k)
        assert np.array_equal(ns.cpu().numpy(), nsel) and np.array_equal(bp.cpu().numpy(), pos)
        assert np.array_equal(bd.cpu().numpy().astype(np.float64), val, equal_nan=True)


def test_empty_inputs_through_the_binding(hdl):
    """Zero roots; roots that are all empty (no tokens at all); zero
    continuations: every call succeeds and writes what the empty case means."""
    e32 = torch.empty(0, dtype=torch.float32, device="cuda")
    eu8 = torch.empty(0, dtype=torch.uint8, device="cuda")
    bp, ns, bd = hdl.hdl_select_branches(e32, eu8, torch.zeros(1, dtype=torch.int64,
                                                                device="cuda"), 4)
    assert bp.numel() == 0 and ns.numel() == 0
    offs = torch.zeros(6, dtype=torch.int64, device="cuda")          # 5 empty roots
    bp, ns, bd = hdl.hdl_select_branches(e32, eu8, offs, 4)
    assert torch.all(ns == 0) and torch.all(bp == -1) and torch.all(torch.isnan(bd))
    conts = torch.zeros(5, dtype=torch.int32, device="cuda")
    cb = hdl.hdl_assign_continuations(ns, bp, conts, n_cont=0)
    assert cb.numel() == 0
    m = hdl.hdl_suffix_mask(cb, torch.zeros(1, dtype=torch.int64, device="cuda"), None,
                            mask_len=0)
    assert m.numel() == 0
