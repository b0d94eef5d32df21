"""GPU top-k selector (selector = 1, through the C ABI) versus the oracle's
selector (oracle/elsaa_oracle.c, steps 1-4 of the selector reading).

The selected key set of every checked query (elsaa_forward_selected_keys)
must equal the oracle's exactly: both sides score keys with the same fp32
chain and break ties by the lower index. O within max-abs 1e-4 (fp32
inputs) / 2e-2 (bf16 inputs) with the relative error reported, log d_s,
d_lr and m as in the sorted-block parity tests.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2607_20214_gb300 import build, elsaa
from paper_2607_20214_gb300.workloads import (WORKLOADS, Workload,
                                              make_gates_lambda, make_inputs)

pytestmark = pytest.mark.gpu

TOL_O = {"fp32": 1e-4, "bf16": 2e-2}
TOL_LOGD = {"fp32": 2e-4, "bf16": 2e-2}
TOL_M = {"fp32": 1e-4, "bf16": 1e-2}
TOL_DLR_REL = {"fp32": 1e-4, "bf16": 1e-2}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    elsaa.load_library()


def run_gpu(wl, x, gates=None, lam=None, **over):
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl, **over)
    xd = {k: v.to(dev) for k, v in x.items()}
    BHN = (wl.B, wl.H, wl.N)
    out = dict(log_d_sparse=torch.full(BHN, float("nan"), device=dev),
               d_lr=torch.full(BHN, float("nan"), device=dev),
               m_sparse=torch.full(BHN, float("nan"), device=dev),
               perm_q=torch.full(BHN, -1, dtype=torch.int32, device=dev),
               perm_k=torch.full(BHN, -1, dtype=torch.int32, device=dev))
    ws = elsaa.new_workspace(p, dev)
    o = elsaa.elsaa_forward(
        p, xd["q"], xd["k"], xd["v"], xd["w_sort"], xd["w_race"],
        lambda_tok=None if lam is None else lam.to(dev),
        gates=None if gates is None else gates.to(dev), workspace=ws, **out)
    keys = elsaa.elsaa_forward_selected_keys(p, ws) if p.selector else None
    elsaa.elsaa_check_status(ws)
    torch.cuda.synchronize()
    res = {k: v.cpu() for k, v in out.items()}
    res["O"] = o.float().cpu()
    res["O_raw"] = o.cpu()
    res["keys"] = None if keys is None else keys.cpu()
    return res


def compare(wl, g, ref, label=""):
    for (b, h), r in ref.items():
        assert np.array_equal(g["perm_q"][b, h].numpy(), r["perm_q"]), label
        assert np.array_equal(g["perm_k"][b, h].numpy(), r["perm_k"]), label
        rows = r["rows"]
        got_sets = g["keys"][b, h].numpy()[rows]
        bad = np.nonzero((got_sets != r["sel"]).any(axis=1))[0]
        assert bad.size == 0, (label, b, h, "key sets differ at rows",
                               rows[bad[:8]])
        O = g["O"][b, h].numpy()[rows]
        err = np.abs(O - r["O"]).max()
        rel = float(np.linalg.norm(O - r["O"]) / np.linalg.norm(r["O"]))
        print("%s head (%d, %d): max |O - O_ref| = %.3e, relative (l2) %.3e"
              % (label, b, h, err, rel))
        assert err <= TOL_O[wl.dtype], (label, b, h, "O", err)
        assert rel <= TOL_O[wl.dtype], (label, b, h, "O relative", rel)
        e = np.abs(g["log_d_sparse"][b, h].numpy()[rows] -
                   r["log_d_sparse"]).max()
        assert e <= TOL_LOGD[wl.dtype], (label, b, h, "log d_s", e)
        dl = g["d_lr"][b, h].numpy()[rows]
        e = (np.abs(dl - r["d_lr"]) / np.abs(r["d_lr"])).max()
        assert e <= TOL_DLR_REL[wl.dtype], (label, b, h, "d_lr", e)
        e = np.abs(g["m_sparse"][b, h].numpy()[rows] - r["m"]).max()
        assert e <= TOL_M[wl.dtype], (label, b, h, "m", e)


def small(dtype="fp32", **kw):
    base = dict(name="topk", B=1, H=2, N=1024, d_h=64, dtype=dtype,
                block=32, race_tables=4, recipe="plain", temperature=2.0,
                seed=31, plane_seed=1031, selector=1, topk=32, topk_blocks=2)
    base.update(kw)
    return Workload(**base)


def oracle(wl, x, heads=None, rows=None, **kw):
    return orc.forward(x, orc.params_from_workload(wl), heads=heads,
                       rows=rows, **kw)


@pytest.mark.parametrize("dtype,d_h,b,c,k", [
    ("fp32", 64, 32, 2, 32), ("fp32", 64, 32, 3, 20), ("fp32", 32, 64, 2, 77),
    ("bf16", 64, 64, 2, 64), ("bf16", 128, 128, 2, 128),
    ("bf16", 128, 32, 4, 50), ("fp32", 128, 128, 2, 200),
    ("bf16", 64, 256, 2, 300), ("bf16", 64, 64, 1, 10),
    ("bf16", 128, 128, 1, 64), ("bf16", 64, 128, 3, 200),
    ("bf16", 128, 256, 1, 100), ("bf16", 64, 128, 4, 128),
])
def test_topk_matches_oracle(dtype, d_h, b, c, k):
    wl = small(dtype, d_h=d_h, block=b, topk_blocks=c, topk=k,
               N=max(1024, 4 * b))
    x = make_inputs(wl)
    compare(wl, run_gpu(wl, x), oracle(wl, x), label=(dtype, d_h, b, c, k))


def test_tensor_core_path_runs_for_bf16_blocks_of_128():
    """bf16 with blocks of 128 or 256 and gamma = 4: the persistent
    tensor-core block kernel walks the candidate blocks (no CUDA-core
    fallback)."""
    wl = small("bf16", d_h=128, block=128, topk_blocks=2, topk=100)
    x = make_inputs(wl)
    elsaa.elsaa_profile_start()
    g = run_gpu(wl, x)
    prof = elsaa.elsaa_profile_stop()
    assert "block_attn_ws" in prof and "block_attn_simt" not in prof, prof
    assert "topk_select" in prof
    compare(wl, g, oracle(wl, x), label="tc path")


def test_topk_ties_on_integer_inputs():
    """Small integer inputs: many exactly equal scores and block scores, so
    the lower-index rule decides a large part of every set."""
    wl = small("fp32", d_h=32, block=32, topk_blocks=3, topk=40, N=512,
               sort_bits=2)
    x = make_inputs(wl)
    for name in ("q", "k"):
        x[name] = torch.round(x[name].clamp(-1.5, 1.5))
    compare(wl, run_gpu(wl, x), oracle(wl, x), label="ties")


def test_one_block_whole_budget_equals_sorted_blocks():
    """c = 1, k = b: every key of the block is kept; the top-k path equals
    the sorted-block path (fp32 on the CUDA cores: the same arithmetic)."""
    wl = small("fp32", topk_blocks=1, topk=32)
    x = make_inputs(wl)
    g = run_gpu(wl, x)
    base = run_gpu(wl.with_(selector=0, topk=0), x)
    assert torch.equal(g["O_raw"], base["O_raw"])
    assert torch.equal(g["log_d_sparse"], base["log_d_sparse"])


def test_topk_gates_lambda_and_fp32_output():
    wl = small("bf16", block=64, topk=48, topk_blocks=2, H=3)
    x = make_inputs(wl)
    gates, lam = make_gates_lambda(wl, seed=9)
    ref = oracle(wl, x, lam=lam, gates=gates)
    g = run_gpu(wl, x, gates=gates, lam=lam, out_fp32=1)
    assert g["O_raw"].dtype == torch.float32
    compare(wl, g, ref, label="gates")


def test_c1_every_row():
    """c1 (B=1 H=1 N=1024 d_h=64 fp32, k=32) with two candidate blocks."""
    wl = WORKLOADS["c1"].with_(selector=1, topk=32, topk_blocks=2)
    x = make_inputs(wl)
    compare(wl, run_gpu(wl, x), oracle(wl, x), label="c1")


def test_c2_six_heads():
    """c2 (B=4 H=12 N=4096 d_h=64 bf16, k=64, planted keys in half the
    heads) with two candidate blocks: six whole heads."""
    wl = WORKLOADS["c2"].with_(selector=1, topk=64, topk_blocks=2)
    x = make_inputs(wl)
    heads = [(0, 0), (0, 1), (1, 6), (2, 3), (3, 10), (3, 11)]
    compare(wl, run_gpu(wl, x), oracle(wl, x, heads=heads), label="c2")


def test_c3_sampled_rows():
    """c3 (B=2 H=16 N=16384 d_h=128 bf16, k=128) with two candidate blocks:
    512 sampled rows of two heads."""
    wl = WORKLOADS["c3"].with_(selector=1, topk=128, topk_blocks=2)
    x = make_inputs(wl)
    rows = np.sort(np.random.default_rng(3).choice(wl.N, 512, replace=False))
    compare(wl, run_gpu(wl, x), oracle(wl, x, heads=[(0, 2), (1, 15)],
                                       rows=rows), label="c3")
