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
