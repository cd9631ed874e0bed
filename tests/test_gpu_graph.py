"""The HDL step (re-scoring, selection, allocation, masks) and the GRPO update
captured in CUDA graphs and replayed give bit for bit what the eager calls
give: every call is capture-safe (kernel launches and one memset, no host
sync)."""
import pytest
import torch

import hdl_synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hdl():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_36864_gb300 as m
    return m


def test_step_in_cuda_graph(hdl):
    spec = hdl_synth.small_spec("graph", n_roots=5, t_lo=100, t_hi=700, d=256, vocab=5000,
                                k=4, conts_per_root=3, seed=17)
    wl = hdl_synth.generate(spec, device="cuda")
    N, R = wl.n_tokens, spec.n_roots
    C = wl.cont_offsets.numel() - 1
    dev = "cuda"
    lp0, lp1, de = (torch.empty(N, device=dev) for _ in range(3))
    ws = torch.empty(hdl.hdl_rescore_workspace_bytes(N, spec.d, spec.vocab), dtype=torch.uint8,
                     device=dev)
    bp = torch.empty((R, spec.k), dtype=torch.int32, device=dev)
    ns = torch.empty(R, dtype=torch.int32, device=dev)
    bd = torch.empty((R, spec.k), device=dev)
    cb = torch.empty(C, dtype=torch.int32, device=dev)
    mask = torch.zeros(wl.cont_valid.numel(), dtype=torch.uint8, device=dev)

    def step(stream):
        hdl.hdl_rescore(wl.h_orig, wl.h_hind, wl.w, wl.targets, lp0, lp1, de, ws, stream=stream)
        hdl.hdl_select_branches(de, wl.valid, wl.root_offsets, spec.k, branch_pos=bp,
                                n_selected=ns, branch_delta=bd, stream=stream)
        hdl.hdl_assign_continuations(ns, bp, wl.conts_per_root, cont_branch=cb, stream=stream)
        hdl.hdl_suffix_mask(cb, wl.cont_offsets, wl.cont_valid, mask=mask, stream=stream)

    step(torch.cuda.current_stream())
    torch.cuda.synchronize()
    eager = [t.clone() for t in (lp0, lp1, de, bp, ns, bd, cb, mask)]
    for t in (lp0, lp1, de, bd):
        t.fill_(float("nan"))
    for t in (bp, ns, cb, mask):
        t.fill_(0)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(g, stream=side):
            step(side)
    torch.cuda.current_stream().wait_stream(side)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    assert hdl.hdl_device_status(ws)[0] == hdl.HDL_OK
    for a, b in zip(eager, (lp0, lp1, de, bp, ns, bd, cb, mask)):
        assert torch.equal(a, b) or torch.equal(torch.nan_to_num(a, nan=-7), torch.nan_to_num(b, nan=-7))


@pytest.mark.parametrize("J,L", [(16, 3000), (12000, 40)])   # the flat and the per-trajectory pass
def test_grpo_in_cuda_graph(hdl, J, L):
    """The GRPO update captured in a CUDA graph and replayed several times
    gives the eager call's advantages, gradient and statistics bit for bit
    (its completion counter is re-armed by the first kernel of every replay)."""
    g = torch.Generator(device="cuda").manual_seed(J)
    T = J * L
    lpo = -torch.rand(T, generator=g, device="cuda") * 3
    lpn = lpo + torch.randn(T, generator=g, device="cuda") * 0.3
    m = (torch.rand(T, generator=g, device="cuda") < 0.7).to(torch.uint8)
    toffs = torch.arange(0, T + 1, L, dtype=torch.int64, device="cuda")
    R = torch.rand(J, generator=g, device="cuda")
    goffs = torch.arange(0, J + 1, 16, dtype=torch.int32, device="cuda")
    adv = torch.empty(J, device="cuda")
    grad = torch.empty(T, device="cuda")
    st = torch.empty(4, device="cuda")
    ws = torch.empty(hdl.hdl_grpo_loss_workspace_bytes(), dtype=torch.uint8, device="cuda")

    def call(stream):
        hdl.hdl_grpo_loss(lpn, lpo, m, toffs, R, goffs, advantages=adv, grad=grad, stats=st,
                          workspace=ws, stream=stream)

    call(torch.cuda.current_stream())
    torch.cuda.synchronize()
    eager = [t.clone() for t in (adv, grad, st)]
    for t in (adv, grad, st):
        t.fill_(float("nan"))
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(graph, stream=side):
            call(side)
    torch.cuda.current_stream().wait_stream(side)
    for _ in range(4):
        graph.replay()
    torch.cuda.synchronize()
    for a, b in zip(eager, (adv, grad, st)):
        assert torch.equal(a, b)
