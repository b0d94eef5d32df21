"""Failure detection without a GPU fault: every wait in the kernels is
bounded; one that runs out records {code, site, CTA} in the workspace status
word and lets its kernel return, so the context stays usable. The self-test
kernel waits on an mbarrier that nothing arrives on; the host reads the
recorded timeout, then runs a normal forward on the same workspace."""
import time

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2607_20214_gb300 import build, elsaa
from paper_2607_20214_gb300.workloads import Workload, make_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    elsaa.load_library()


def test_bounded_wait_timeout_is_reported_and_context_survives():
    wl = Workload(name="fail", B=1, H=2, N=512, d_h=64, dtype="bf16",
                  block=64, race_tables=4, recipe="plain", temperature=2.0,
                  seed=41, plane_seed=1041)
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl)
    ws = elsaa.new_workspace(p, dev)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    elsaa.elsaa_selftest_wait_timeout(ws, limit_ms=100)
    with pytest.raises(elsaa.ElsaaError) as e:
        elsaa.elsaa_check_status(ws)
    elapsed = time.perf_counter() - t0
    assert e.value.code == elsaa.ELSAA_ERR_DEVICE
    assert "status 3" in str(e.value)          # kDevWaitTimeout
    assert "site %d" % 0x7E57 in str(e.value)  # the self-test's wait
    assert 0.1 <= elapsed < 10.0               # it waited, then gave up
    # the context is intact: a forward on the same workspace clears the
    # status word and matches the oracle
    x = make_inputs(wl)
    xd = {k: v.to(dev) for k, v in x.items()}
    o = elsaa.elsaa_forward(p, xd["q"], xd["k"], xd["v"], xd["w_sort"],
                            xd["w_race"], workspace=ws)
    elsaa.elsaa_check_status(ws)
    ref = orc.forward(x, orc.params_from_workload(wl), heads=[(0, 1)])
    err = np.abs(o[0, 1].float().cpu().numpy() - ref[(0, 1)]["O"]).max()
    assert err <= 2e-2


@pytest.mark.parametrize("dtype,impl", [("bf16", elsaa.ELSAA_IMPL_AUTO),
                                        ("fp32", elsaa.ELSAA_IMPL_SIMT)])
def test_bad_permutation_entry_is_reported_not_read(dtype, impl):
    """elsaa_backward takes the sort orders from its caller. An entry
    outside [0, N) is recorded in the status word (code 2, permutation
    range) and read as row 0 instead of reaching memory out of bounds, on
    the tensor-core and the CUDA-core backward; a call with the correct
    orders afterwards is clean."""
    wl = Workload(name="perm", B=1, H=2, N=512, d_h=64, dtype=dtype,
                  block=64, race_tables=8, recipe="plain", temperature=2.0,
                  seed=43, plane_seed=1043, backward=True)
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl, impl=impl)
    x = {k: v.to(dev) for k, v in make_inputs(wl).items()}
    BHN = (wl.B, wl.H, wl.N)
    pq = torch.empty(BHN, dtype=torch.int32, device=dev)
    pk = torch.empty(BHN, dtype=torch.int32, device=dev)
    elsaa.elsaa_forward(p, x["q"], x["k"], x["v"], x["w_sort"], x["w_race"],
                        perm_q=pq, perm_k=pk)
    bad_q, bad_k = pq.clone(), pk.clone()
    bad_q[0, 1, 7] = wl.N + 7
    bad_k[0, 0, 100] = -3
    n = elsaa.elsaa_backward_workspace_size(p)
    ws = torch.empty(max(n, 256), dtype=torch.uint8, device=dev)
    elsaa.elsaa_backward(p, x["q"], x["k"], x["v"], x["w_sort"], x["w_race"],
                         x["do"], bad_q, bad_k, workspace=ws)
    with pytest.raises(elsaa.ElsaaError) as e:
        elsaa.elsaa_check_status(ws)
    assert e.value.code == elsaa.ELSAA_ERR_DEVICE
    assert "status 2" in str(e.value)
    dq, dk, dv = elsaa.elsaa_backward(p, x["q"], x["k"], x["v"], x["w_sort"],
                                      x["w_race"], x["do"], pq, pk,
                                      workspace=ws)
    elsaa.elsaa_check_status(ws)
    assert torch.isfinite(dq).all() and torch.isfinite(dv).all()
