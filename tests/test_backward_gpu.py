"""GPU backward (elsaa_backward through the C ABI) versus the oracle's
analytic fp64 gradient on the same seeded inputs.

The permutations come from the GPU forward and must equal the oracle's
(integer work, bit-exact). Gradients are compared relative to the largest
reference magnitude of each tensor, by their relative l2 error, and row by
row: the relative l2 error of each row on its own scale, 99 % of rows
within five times the bound (the others are rows whose terms cancel
under the softmax gradient: such a row is far smaller than its terms, and
so than their rounding errors). The CUDA-core path keeps every operand
in fp32 and accumulates over at most b + r terms per element (b <= 128,
r <= 256): its error stays near 1e-6 of that magnitude; its bound is 1e-3.
The tensor-core path (bf16 inputs, b = 64, d_h = 64) rounds its MMA
operands (E, dZ, X, gNum, phi, dL/du and the B summary) to bf16, a relative
2^-9 = 2e-3 per operand, with fp32 accumulation: errors of a few 1e-3 of
the largest magnitude; its bound is 1e-2. Which path ran is read from the
library's per-kernel profile.
"""
import numpy as np
import pytest
import torch

from oracle import backward as bwd
from oracle import oracle as orc
from paper_2607_20214_gb300 import build, elsaa
from paper_2607_20214_gb300.workloads import (WORKLOADS, Workload,
                                              make_gates_lambda, make_inputs)

pytestmark = pytest.mark.gpu

TOL_REL = 1e-3     # CUDA-core backward (fp32 operands)
TOL_REL_TC = 1e-2  # tensor-core backward (bf16 operands)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    elsaa.load_library()


def run_gpu(wl, x, gates=None, lam=None, impl=elsaa.ELSAA_IMPL_AUTO):
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl, impl=impl)
    xd = {k: v.to(dev) for k, v in x.items()}
    BHN = (wl.B, wl.H, wl.N)
    perm_q = torch.empty(BHN, dtype=torch.int32, device=dev)
    perm_k = torch.empty(BHN, dtype=torch.int32, device=dev)
    g = None if gates is None else gates.to(dev)
    lt = None if lam is None else lam.to(dev)
    elsaa.elsaa_forward(p, xd["q"], xd["k"], xd["v"], xd["w_sort"],
                        xd["w_race"], lambda_tok=lt, gates=g,
                        perm_q=perm_q, perm_k=perm_k)
    d_gates = torch.full(BHN + (2,), float("nan"), device=dev)
    d_lambda = torch.full(BHN, float("nan"), device=dev)
    torch.cuda.synchronize()
    elsaa.elsaa_profile_start()
    dq, dk, dv = elsaa.elsaa_backward(
        p, xd["q"], xd["k"], xd["v"], xd["w_sort"], xd["w_race"], xd["do"],
        perm_q, perm_k, lambda_tok=lt, gates=g, d_gates=d_gates,
        d_lambda=d_lambda)
    prof = elsaa.elsaa_profile_stop()
    torch.cuda.synchronize()
    return dict(dQ=dq.cpu(), dK=dk.cpu(), dV=dv.cpu(),
                dgates=d_gates.cpu(), dlam=d_lambda.cpu(),
                perm_q=perm_q.cpu(), perm_k=perm_k.cpu(),
                tc="bwd_block_tc" in prof)


@pytest.mark.parametrize("impl,dtype", [(elsaa.ELSAA_IMPL_AUTO, "bf16"),
                                        (elsaa.ELSAA_IMPL_SIMT, "fp32")])
def test_saved_race_summaries_match_recompute(impl, dtype):
    """elsaa_backward with the forward's A, B (elsaa_forward_race_summaries)
    gives the same gradients, bit for bit, as with A, B recomputed; and the
    saved summaries equal the oracle's to rounding."""
    wl = small(dtype, N=1024, race_tables=8)
    x = make_inputs(wl)
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl, impl=impl)
    xd = {k: v.to(dev) for k, v in x.items()}
    BHN = (wl.B, wl.H, wl.N)
    perm_q = torch.empty(BHN, dtype=torch.int32, device=dev)
    perm_k = torch.empty(BHN, dtype=torch.int32, device=dev)
    ws = elsaa.new_workspace(p, dev)
    elsaa.elsaa_forward(p, xd["q"], xd["k"], xd["v"], xd["w_sort"],
                        xd["w_race"], perm_q=perm_q, perm_k=perm_k,
                        workspace=ws)
    A, B = elsaa.elsaa_forward_race_summaries(p, ws)
    args = (p, xd["q"], xd["k"], xd["v"], xd["w_sort"], xd["w_race"],
            xd["do"], perm_q, perm_k)
    g0 = elsaa.elsaa_backward(*args)
    g1 = elsaa.elsaa_backward(*args, race_A=A, race_B=B)
    torch.cuda.synchronize()
    for a, c in zip(g0, g1):
        assert torch.equal(a, c)
    # the saved summaries are the forward's A, B (Algorithm RACE steps 5-7)
    for h in range(wl.H):
        Ar, Br = orc.race_summaries(x["k"][0, h].double().numpy(),
                                    x["v"][0, h].double().numpy(),
                                    x["w_race"][h].double().numpy(), wl.beta)
        Ag = A[0, h].cpu().double().numpy().reshape(Ar.shape)
        Bg = B[0, h].cpu().double().numpy().reshape(Br.shape)
        tol = 1e-2 if dtype == "bf16" else 1e-4
        assert np.abs(Ag - Ar).max() <= tol * np.abs(Ar).max()
        assert np.abs(Bg - Br).max() <= tol * np.abs(Br).max()


def oracle_head(wl, x, b, h, gates=None, lam=None):
    f32 = lambda t: t[b, h].float().cpu().numpy()
    p = orc.params_from_workload(wl)
    lam_h = None if lam is None else lam[b, h].double().numpy()
    gates_h = None if gates is None else gates[b, h].double().numpy()
    if lam_h is None:
        lam_h = np.full(wl.N, wl.lam)
    return bwd.backward_head(
        f32(x["q"]), f32(x["k"]), f32(x["v"]),
        x["w_sort"][h].float().cpu().numpy(),
        x["w_race"][h].double().cpu().numpy(), f32(x["do"]), p, lam=lam_h,
        gates=gates_h)


def compare(wl, g, x, heads, gates=None, lam=None):
    tol = TOL_REL_TC if g["tc"] else TOL_REL
    worst = {}
    for (b, h) in heads:
        r = oracle_head(wl, x, b, h, gates, lam)
        assert np.array_equal(g["perm_q"][b, h].numpy(), r["perm_q"])
        assert np.array_equal(g["perm_k"][b, h].numpy(), r["perm_k"])
        for name in ("dQ", "dK", "dV"):
            ref = r[name]
            got = g[name][b, h].numpy().astype(np.float64)
            err = np.abs(got - ref).max() / np.abs(ref).max()
            worst[name] = max(worst.get(name, 0.0), err)
            assert err <= tol, (name, b, h, err)
            # spread-out errors: relative l2 over the tensor, and per row
            # (a row on its own scale, so small-magnitude rows are checked
            # too) for all but the 1 % of rows where the softmax gradient's
            # cancellation leaves the row much smaller than its terms
            l2 = np.linalg.norm(got - ref) / np.linalg.norm(ref)
            assert l2 <= tol, (name, b, h, "rel l2", l2)
            rn = np.linalg.norm(ref, axis=1)
            live = rn > 0
            rows = np.linalg.norm(got - ref, axis=1)[live] / rn[live]
            q99 = np.quantile(rows, 0.99)
            assert q99 <= 5 * tol, (name, b, h, "row rel l2 p99", q99)
        ref = r["dgates"]
        err = np.abs(g["dgates"][b, h].numpy() - ref).max() / np.abs(ref).max()
        assert err <= tol, ("dgates", b, h, err)
        if wl.fusion_mode == 0:
            ref = r["dlam"]
            err = (np.abs(g["dlam"][b, h].numpy() - ref).max()
                   / max(np.abs(ref).max(), 1e-30))
            assert err <= tol, ("dlam", b, h, err)
    return worst


def small(dtype="bf16", **kw):
    base = dict(name="small", B=1, H=2, N=384, d_h=64, dtype=dtype, block=64,
                race_tables=4, recipe="plain", temperature=2.0, seed=21,
                plane_seed=1021, backward=True)
    base.update(kw)
    return Workload(**base)


@pytest.mark.parametrize("dtype,impl,tc", [
    ("fp32", elsaa.ELSAA_IMPL_AUTO, False),
    ("bf16", elsaa.ELSAA_IMPL_AUTO, True),
    ("bf16", elsaa.ELSAA_IMPL_SIMT, False)])
def test_small_backward_matches_oracle(dtype, impl, tc):
    wl = small(dtype)
    x = make_inputs(wl)
    gates, lam = make_gates_lambda(wl, seed=3)
    g = run_gpu(wl, x, gates, lam, impl=impl)
    assert g["tc"] == tc  # the path that was meant to run did
    compare(wl, g, x, [(0, 0), (0, 1)], gates, lam)


def test_tensor_core_backward_shapes():
    """The tensor-core path's shape class: L_s = 8 (r = 128, the c5 setting),
    several head-major tiles per CTA, the m = 1 ablation."""
    for over in (dict(race_tables=8, N=1024, H=3),
                 dict(race_tables=8, fusion_mode=1)):
        wl = small("bf16").with_(**over)
        x = make_inputs(wl)
        g = run_gpu(wl, x)
        assert g["tc"]
        compare(wl, g, x, [(0, 0), (0, wl.H - 1)])


@pytest.mark.parametrize("L", [4, 8])
def test_tensor_core_backward_several_tiles_per_cta(L):
    """260 tiles (26 per head) over the 152 persistent CTAs: 108 CTAs take
    two tiles, four of them across a head change (tiles 25-26, 51-52,
    155-156, 181-182), so the second Q/K buffer, the planes kept per
    buffer, the per-head sums reloaded mid-CTA and the bucket-sum partials
    of a head split over several CTAs are all exercised; every head is
    compared."""
    wl = small("bf16", H=10, N=3328, race_tables=L, seed=31 + L)
    x = make_inputs(wl)
    gates, lam = make_gates_lambda(wl, seed=5) if L == 8 else (None, None)
    g = run_gpu(wl, x, gates, lam)
    assert g["tc"]
    compare(wl, g, x, [(0, h) for h in range(wl.H)], gates, lam)


@pytest.mark.parametrize("over", [dict(fusion_mode=1), dict(block=32),
                                  dict(d_h=32, race_bits=3, race_tables=6),
                                  dict(block=128, d_h=32, race_tables=2)])
def test_backward_variants(over):
    wl = small("bf16").with_(**over)
    x = make_inputs(wl)
    compare(wl, run_gpu(wl, x), x, [(0, 0), (0, 1)])


def test_c5_full_size_sampled_heads():
    """The training workload at full size (96 heads); the oracle checks
    two whole heads."""
    wl = WORKLOADS["c5"]
    x = make_inputs(wl, device="cuda")
    g = run_gpu(wl, x)
    assert g["tc"]
    xc = {k: v.cpu() for k, v in x.items()}
    compare(wl, g, xc, [(0, 0), (7, 11)])


def test_backward_cuda_graph_with_saved_summaries():
    """elsaa_backward with saved A, B captured into a CUDA graph and
    replayed: bit-identical to an eager call."""
    wl = small("bf16", N=1024, race_tables=8)
    x = make_inputs(wl)
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl)
    xd = {k: v.to(dev) for k, v in x.items()}
    BHN = (wl.B, wl.H, wl.N)
    perm_q = torch.empty(BHN, dtype=torch.int32, device=dev)
    perm_k = torch.empty(BHN, dtype=torch.int32, device=dev)
    ws = elsaa.new_workspace(p, dev)
    st = torch.cuda.Stream(dev)
    with torch.cuda.stream(st):
        elsaa.elsaa_forward(p, xd["q"], xd["k"], xd["v"], xd["w_sort"],
                            xd["w_race"], perm_q=perm_q, perm_k=perm_k,
                            workspace=ws, stream=st)
        A, B = elsaa.elsaa_forward_race_summaries(p, ws, stream=st)
    wsb = torch.empty(elsaa.elsaa_backward_workspace_size(p),
                      dtype=torch.uint8, device=dev)
    grads = [torch.empty(xd["q"].shape, dtype=torch.float32, device=dev)
             for _ in range(3)]

    def call():
        elsaa.elsaa_backward(p, xd["q"], xd["k"], xd["v"], xd["w_sort"],
                             xd["w_race"], xd["do"], perm_q, perm_k,
                             dq=grads[0], dk=grads[1], dv=grads[2],
                             race_A=A, race_B=B, workspace=wsb, stream=st)

    with torch.cuda.stream(st):
        call()
    st.synchronize()
    eager = [g.clone() for g in grads]
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=st):
        call()
    for g in grads:
        g.zero_()
    graph.replay()
    torch.cuda.synchronize()
    elsaa.elsaa_check_status(wsb)
    for a, b in zip(eager, grads):
        assert torch.equal(a, b)
