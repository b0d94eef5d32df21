"""The checked build (libelsaa_checked.so, ELSAA_CHECKED): the forward
kernels also record permutation entries outside [0, N) in the status word
(the default build reads them as row 0 without recording, because the
check costs 4 % of the block kernel and the forward's orders come from its
own sort). The checked library must compute exactly what the default one
computes, report nothing on valid inputs, and report a bad caller-supplied
order (the backward takes its orders from the caller).
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2607_20214_gb300 import build, elsaa
from paper_2607_20214_gb300.workloads import Workload, make_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def checked():
    """Swaps the checked library in for the module's tests."""
    build.build()
    path = build.build_checked()
    saved = elsaa.load_library()
    elsaa._lib = None
    lib = elsaa.load_library(path)
    yield lib
    elsaa._lib = saved


def _forward(lib_swap, wl, x, **over):
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl, **over)
    xd = {k: v.to(dev) for k, v in x.items()}
    ws = elsaa.new_workspace(p, dev)
    o = elsaa.elsaa_forward(p, xd["q"], xd["k"], xd["v"], xd["w_sort"],
                            xd["w_race"], workspace=ws)
    elsaa.elsaa_check_status(ws)
    return o.cpu()


@pytest.mark.parametrize("causal,block", [(0, 128), (1, 128), (0, 256)])
def test_checked_build_computes_the_same(checked, causal, block):
    """block 256: the CTA-pair kernel."""
    wl = Workload(name="chk", B=1, H=2, N=1024, d_h=128, dtype="bf16",
                  block=block, race_tables=16, recipe="plain",
                  temperature=2.0, seed=51, plane_seed=1051, causal=causal,
                  causal_base_len=256)
    x = make_inputs(wl)
    got = _forward(checked, wl, x)
    # the default library on the same inputs
    lib_checked = elsaa._lib
    elsaa._lib = None
    elsaa.load_library(build.LIB)
    try:
        want = _forward(None, wl, x)
    finally:
        elsaa._lib = lib_checked
    assert torch.equal(got, want)
    if not causal:
        ref = orc.forward(x, orc.params_from_workload(wl))
        for (b, h), r in ref.items():
            assert np.abs(got[b, h].float().numpy() - r["O"]).max() <= 2e-2


def test_checked_build_reports_a_bad_order(checked):
    wl = Workload(name="chk", B=1, H=2, N=512, d_h=64, dtype="bf16",
                  block=64, race_tables=8, recipe="plain", temperature=2.0,
                  seed=53, plane_seed=1053, backward=True)
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl)
    x = {k: v.to(dev) for k, v in make_inputs(wl).items()}
    BHN = (wl.B, wl.H, wl.N)
    pq = torch.empty(BHN, dtype=torch.int32, device=dev)
    pk = torch.empty(BHN, dtype=torch.int32, device=dev)
    elsaa.elsaa_forward(p, x["q"], x["k"], x["v"], x["w_sort"], x["w_race"],
                        perm_q=pq, perm_k=pk)
    bad = pq.clone()
    bad[0, 0, 3] = -1
    n = elsaa.elsaa_backward_workspace_size(p)
    ws = torch.empty(max(n, 256), dtype=torch.uint8, device=dev)
    elsaa.elsaa_backward(p, x["q"], x["k"], x["v"], x["w_sort"], x["w_race"],
                         x["do"], bad, pk, workspace=ws)
    with pytest.raises(elsaa.ElsaaError) as e:
        elsaa.elsaa_check_status(ws)
    assert "status 2" in str(e.value)
