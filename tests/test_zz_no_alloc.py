"""elsaa_forward_noalloc: the forward pass for callers that cannot allocate
device memory (for example a plug-in whose host application owns all device
buffers and offers no allocator, or a path that must not risk the
device-wide synchronisation of cudaMalloc / cudaFree). Its scratch is a fixed
array inside the library, shared by every call, so these checks compare it
with elsaa_forward (caller-provided workspace) on calls in a row, including a
larger problem followed by a smaller one of another shape (stale scratch from
the first must not reach the second), read its status word through
elsaa_check_status_noalloc, and check that a problem larger than the array is
refused.

This file is named so that pytest collects it last.
"""
import ctypes
import time

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2607_20214_gb300 import build, elsaa
from paper_2607_20214_gb300.workloads import Workload, make_inputs

pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-4, "bf16": 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    elsaa.load_library()


def _case(dtype, N=1184, block=32, seed=21, d_h=64, race_tables=4):
    return Workload("noalloc", B=2, H=2, N=N, d_h=d_h, dtype=dtype,
                    block=block, race_tables=race_tables, recipe="plain",
                    temperature=2.0, seed=seed, plane_seed=1000 + seed)


def _compare(wl, dev):
    """One elsaa_forward_noalloc call against elsaa_forward on the same
    inputs: O within the dtype's bound, both sort orders identical."""
    dtype = wl.dtype
    x = {k: t.to(dev) for k, t in make_inputs(wl).items()}
    p = elsaa.params_for(wl)
    assert elsaa.elsaa_workspace_size(p) <= \
        elsaa.ELSAA_STATIC_WORKSPACE_BYTES
    BHN = (wl.B, wl.H, wl.N)
    ref_pq = torch.empty(BHN, dtype=torch.int32, device=dev)
    ref_pk = torch.empty(BHN, dtype=torch.int32, device=dev)
    ref = elsaa.elsaa_forward(p, x["q"], x["k"], x["v"], x["w_sort"],
                              x["w_race"], perm_q=ref_pq, perm_k=ref_pk)
    torch.cuda.synchronize()
    o = torch.full_like(x["q"], float("nan"))
    pq = torch.full(BHN, -1, dtype=torch.int32, device=dev)
    pk = torch.full(BHN, -1, dtype=torch.int32, device=dev)
    elsaa.elsaa_forward_noalloc(p, x["q"], x["k"], x["v"], x["w_sort"],
                                x["w_race"], o=o, perm_q=pq, perm_k=pk)
    elsaa.elsaa_check_status_noalloc()
    err = (o.float() - ref.float()).abs().max().item()
    assert err <= TOL[dtype], err
    assert torch.equal(pq, ref_pq)
    assert torch.equal(pk, ref_pk)


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_noalloc_matches_workspace_entry_point_twice(dtype):
    dev = torch.device("cuda:0")
    for _ in range(2):
        _compare(_case(dtype), dev)


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_noalloc_larger_then_smaller_problem(dtype):
    """The shared array keeps the previous call's contents: a smaller call
    of another N and block size after a larger one must match the
    workspace entry point exactly in its sort orders."""
    dev = torch.device("cuda:0")
    _compare(_case(dtype, N=4096, block=64, seed=23), dev)
    _compare(_case(dtype, N=1184, block=32, seed=24), dev)


def test_noalloc_tensor_core_kernels():
    """bf16 shapes that take the one-CTA tensor-core block kernel (b = 128)
    and the CTA-pair kernel (b = 256, d_h = 128) through the static array."""
    dev = torch.device("cuda:0")
    _compare(_case("bf16", N=2048, block=128, seed=25, d_h=128,
                   race_tables=16), dev)
    _compare(_case("bf16", N=2048, block=256, seed=26, d_h=128,
                   race_tables=16), dev)


def test_noalloc_status_word_reports_timeout_then_clears():
    """The static array's status word is readable without its address: the
    bounded-wait self-test records a timeout there, and the next forward
    clears it and matches the oracle."""
    dev = torch.device("cuda:0")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    elsaa.elsaa_selftest_wait_timeout_noalloc(limit_ms=100)
    with pytest.raises(elsaa.ElsaaError) as e:
        elsaa.elsaa_check_status_noalloc()
    assert time.perf_counter() - t0 >= 0.1
    assert e.value.code == elsaa.ELSAA_ERR_DEVICE
    assert "status 3" in str(e.value)
    assert "site %d" % 0x7E57 in str(e.value)
    wl = _case("bf16", seed=25)
    x = make_inputs(wl)
    xd = {k: v.to(dev) for k, v in x.items()}
    o = torch.empty_like(xd["q"])
    elsaa.elsaa_forward_noalloc(elsaa.params_for(wl), xd["q"], xd["k"],
                                xd["v"], xd["w_sort"], xd["w_race"], o=o)
    elsaa.elsaa_check_status_noalloc()
    ref = orc.forward(x, orc.params_from_workload(wl), heads=[(1, 0)])
    err = np.abs(o[1, 0].float().cpu().numpy() - ref[(1, 0)]["O"]).max()
    assert err <= TOL["bf16"]


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
