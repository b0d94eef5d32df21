"""elsaa_forward_noalloc: the forward pass for callers that cannot allocate
device memory (for example a plug-in whose host application owns all device
buffers and offers no allocator, or a path that must not risk the
device-wide synchronisation of cudaMalloc / cudaFree). Its scratch is a fixed
array inside the library, so these checks compare it with elsaa_forward
(caller-provided workspace) on two calls in a row, and check that a problem
larger than the array is refused.

This file is named so that pytest collects it last.
"""
import ctypes

import pytest
import torch

from paper_2607_20214_gb300 import build, elsaa
from paper_2607_20214_gb300.workloads import Workload, make_inputs

pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-4, "bf16": 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    elsaa.load_library()


def _case(dtype):
    return Workload("noalloc", B=2, H=2, N=1184, d_h=64, dtype=dtype,
                    block=32, race_tables=4, recipe="plain", temperature=2.0,
                    seed=21, plane_seed=1021)


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_noalloc_matches_workspace_entry_point_twice(dtype):
    wl = _case(dtype)
    dev = torch.device("cuda:0")
    x = {k: t.to(dev) for k, t in make_inputs(wl).items()}
    p = elsaa.params_for(wl)
    assert elsaa.elsaa_workspace_size(p) <= \
        elsaa.ELSAA_STATIC_WORKSPACE_BYTES
    BHN = (wl.B, wl.H, wl.N)
    ref_perm = torch.empty(BHN, dtype=torch.int32, device=dev)
    ref = elsaa.elsaa_forward(p, x["q"], x["k"], x["v"], x["w_sort"],
                              x["w_race"], perm_q=ref_perm)
    torch.cuda.synchronize()
    for call in range(2):
        o = torch.full_like(x["q"], float("nan"))
        perm = torch.full(BHN, -1, dtype=torch.int32, device=dev)
        elsaa.elsaa_forward_noalloc(p, x["q"], x["k"], x["v"], x["w_sort"],
                                    x["w_race"], o=o, perm_q=perm)
        torch.cuda.synchronize()
        err = (o.float() - ref.float()).abs().max().item()
        assert err <= TOL[dtype], (call, err)
        assert torch.equal(perm, ref_perm), call


def test_noalloc_refuses_problem_larger_than_its_array():
    lib = elsaa.load_library()
    p = elsaa.make_params(B=4, H=32, N=65536, d_h=128, block_size=256,
                          race_tables=16)
    assert elsaa.elsaa_workspace_size(p) > elsaa.ELSAA_STATIC_WORKSPACE_BYTES
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: rejected first
    rc = lib.elsaa_forward_noalloc(ctypes.byref(p), fake, fake, fake, fake,
                                   fake, None, None, fake, None, None, None,
                                   None, None, None)
    assert rc == elsaa.ELSAA_ERR_WORKSPACE
    assert "static array" in elsaa.elsaa_last_error()
