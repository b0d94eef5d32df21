"""GPU causal path (elsaa_forward with causal = 1, through the C ABI) versus
the fp64 causal oracle (oracle/causal.py) on the same seeded inputs.

Selection: the sorted orders of every SortLSH call of the recursion
(elsaa_causal_index_lists: each node's future-half queries and past-half
keys, stably sorted by code) equal the oracle's orders exactly, at every
level. They fix which keys every query attends.

Outputs: the operator is checked with an fp32 output (out_fp32 = 1), O
within max-abs 2e-2 of the oracle (the bf16-input bound: the kernels round
the softmax weights, the RACE features, the masked intra-chunk products and
the prefix states sB_n to bf16 before their tensor-core products and
accumulate in fp32); the relative error ||O - O_ref|| / ||O_ref|| is
reported beside it. A bf16 output must equal the fp32 output rounded to
bf16 (round to nearest even): the same arithmetic, rounded once at the
store. Causal rows near the start average over a handful of keys, so |O|
reaches 5-8 there, where a bf16 ulp is 2^-5; that rounding alone can exceed
2e-2, so bf16 outputs are compared with the oracle within 2e-2 plus half a
bf16 ulp of |O_ref|. log d_sparse within 2e-2 absolute (fp32 running
maximum and sum), d_lr within 1e-2 relative, m within 1e-2 absolute.
"""
import numpy as np
import pytest
import torch

from oracle import causal as oc
from oracle import oracle as orc
from paper_2607_20214_gb300 import build, elsaa
from paper_2607_20214_gb300.workloads import (WORKLOADS, Workload,
                                              make_gates_lambda, make_inputs)

pytestmark = pytest.mark.gpu

TOL_O, TOL_LOGD, TOL_DLR_REL, TOL_M = 2e-2, 2e-2, 1e-2, 1e-2
HALF_ULP_BF16 = 2.0 ** -8  # relative


def o_err(got, ref):
    """Largest error of a bf16 O in units of its bound 2e-2 + 2^-8 |O_ref|."""
    return (np.abs(got - ref) / (TOL_O + HALF_ULP_BF16 * np.abs(ref))).max()


def rel_l2(got, ref):
    return float(np.linalg.norm(got - ref) / np.linalg.norm(ref))


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    elsaa.load_library()


def run_gpu(wl, x, gates=None, lam=None, out_fp32=0):
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl, out_fp32=out_fp32)
    xd = {k: v.to(dev) for k, v in x.items()}
    BHN = (wl.B, wl.H, wl.N)
    out = dict(log_d_sparse=torch.full(BHN, float("nan"), device=dev),
               d_lr=torch.full(BHN, float("nan"), device=dev),
               m_sparse=torch.full(BHN, float("nan"), device=dev))
    ws = elsaa.new_workspace(p, dev)
    o = elsaa.elsaa_forward(
        p, xd["q"], xd["k"], xd["v"], xd["w_sort"], xd["w_race"],
        lambda_tok=None if lam is None else lam.to(dev),
        gates=None if gates is None else gates.to(dev), workspace=ws, **out)
    lists = elsaa.elsaa_causal_index_lists(p, ws)
    elsaa.elsaa_check_status(ws)
    torch.cuda.synchronize()
    res = {k: v.cpu() for k, v in out.items()}
    res["O"] = o.float().cpu()
    res["O_raw"] = o.cpu()
    res["lists"] = None if lists is None else lists.cpu().numpy()
    return res


def compare_lists(g, ref, label=""):
    """The SortLSH orders of every level, bit-exact."""
    for (b, h), r in ref.items():
        want = r["index_lists"]
        if g["lists"] is None:
            assert not want, (label, "levels")
            continue
        assert g["lists"].shape[0] == len(want), (label, "levels")
        for level, (qrows, krows) in want.items():
            assert np.array_equal(g["lists"][level - 1, 0, b, h], qrows), \
                (label, b, h, level, "query order")
            assert np.array_equal(g["lists"][level - 1, 1, b, h], krows), \
                (label, b, h, level, "key order")


def compare(g, ref, label="", fp32_out=False):
    compare_lists(g, ref, label)
    for (b, h), r in ref.items():
        got = g["O"][b, h].numpy()
        if fp32_out:
            e = np.abs(got - r["O"]).max()
            rel = rel_l2(got, r["O"])
            print("%s head (%d, %d): max |O - O_ref| = %.3e, relative "
                  "(l2) %.3e" % (label, b, h, e, rel))
            assert e <= TOL_O, (label, b, h, "O", e)
            assert rel <= TOL_O, (label, b, h, "O relative", rel)
        else:
            e = o_err(got, r["O"])
            assert e <= 1.0, (label, b, h, "O (in units of its bound)", e)
        e = np.abs(g["log_d_sparse"][b, h].numpy() - r["log_d_sparse"]).max()
        assert e <= TOL_LOGD, (label, b, h, "log d_s", e)
        dl = g["d_lr"][b, h].numpy()
        e = (np.abs(dl - r["d_lr"]) / np.abs(r["d_lr"])).max()
        assert e <= TOL_DLR_REL, (label, b, h, "d_lr", e)
        e = np.abs(g["m_sparse"][b, h].numpy() - r["m_log"]).max()
        assert e <= TOL_M, (label, b, h, "m", e)


def small(**kw):
    base = dict(name="causal", B=1, H=2, N=1024, d_h=64, dtype="bf16",
                block=64, race_tables=8, recipe="plain", temperature=2.0,
                seed=21, plane_seed=1021, causal=1, causal_chunk=128,
                causal_base_len=256)
    base.update(kw)
    return Workload(**base)


def check_bf16_is_rounded_fp32(g16, g32, label=""):
    """The bf16 output is the fp32 output rounded once to bf16."""
    assert torch.equal(g16["O_raw"], g32["O_raw"].to(torch.bfloat16)), label


@pytest.mark.parametrize("d_h,b,L,N,N0,n_s", [
    (64, 64, 8, 1024, 256, 5),      # two levels above 256-row segments
    (128, 128, 16, 1024, 256, 5),
    (128, 256, 16, 2048, 512, 5),   # blocks of two key tiles
    (64, 32, 4, 512, 128, 5),       # four blocks per 128-row tile
    (64, 64, 8, 512, 4096, 5),      # one segment: exact causal attention
    (128, 128, 8, 2048, 300, 5),    # three levels, segments of 256 rows
    (128, 64, 4, 1024, 256, 5),     # r = 64 (one half-filled bucket group)
    (64, 128, 16, 1024, 512, 5),    # r = 256 at d_h = 64 (staged sparse rows)
    (64, 64, 8, 2048, 256, 1),      # two codes: long runs of tied codes
    (128, 128, 16, 1024, 256, 0),   # no sort bits: one code, identity order
])
def test_causal_matches_oracle(d_h, b, L, N, N0, n_s):
    wl = small(d_h=d_h, block=b, race_tables=L, N=N, causal_base_len=N0,
               sort_bits=n_s)
    x = make_inputs(wl)
    ref = oc.forward(x, orc.params_from_workload(wl))
    label = (d_h, b, L, N, N0, n_s)
    g32 = run_gpu(wl, x, out_fp32=1)
    compare(g32, ref, label=label, fp32_out=True)
    g16 = run_gpu(wl, x)
    compare(g16, ref, label=label)
    check_bf16_is_rounded_fp32(g16, g32, label)


def test_causal_duplicate_keys_tie_break():
    """Exact duplicate keys (every 64th key repeated half a sequence later,
    the long-context recipe) share codes: the stable order must keep them
    by increasing index at every level."""
    wl = small(N=2048, recipe="dup_keys", causal_base_len=256)
    x = make_inputs(wl)
    ref = oc.forward(x, orc.params_from_workload(wl))
    compare(run_gpu(wl, x, out_fp32=1), ref, label="dup", fp32_out=True)


def test_causal_gates_lambda_and_ablation():
    wl = small(H=3)
    x = make_inputs(wl)
    gates, lam = make_gates_lambda(wl, seed=5)
    ref = oc.forward(x, orc.params_from_workload(wl), lam=lam, gates=gates)
    compare(run_gpu(wl, x, gates=gates, lam=lam), ref, label="gates")
    wl1 = wl.with_(fusion_mode=1)
    ref = oc.forward(x, orc.params_from_workload(wl1))
    g = run_gpu(wl1, x)
    for (b, h), r in ref.items():
        assert o_err(g["O"][b, h].numpy(), r["O"]) <= 1.0
        assert (g["m_sparse"][b, h].numpy() == 1.0).all()


def test_causal_prefix_rows_ignore_later_keys():
    """Rows before t do not change when keys and values after t change
    (the device path keeps the causal structure)."""
    wl = small(N=1024)
    x = make_inputs(wl)
    a = run_gpu(wl, x)
    y = {k: v.clone() for k, v in x.items()}
    y["k"][:, :, 700:] = -y["k"][:, :, 700:]
    y["v"][:, :, 700:] = 3.0
    c = run_gpu(wl, y)
    assert torch.equal(a["O"][:, :, :700], c["O"][:, :, :700])
    assert (a["O"][:, :, 700:] - c["O"][:, :, 700:]).abs().max() > 0.1


def test_c3_causal_full_size_heads():
    """The c3 causal workload (B=2 H=16 N=16384 d_h=128, b=128, r=256,
    C=128, N_0=4096) in the benchmark's launch configuration; every row of
    two heads against the oracle."""
    wl = WORKLOADS["c3c"]
    x = make_inputs(wl)
    g32 = run_gpu(wl, x, out_fp32=1)
    ref = oc.forward(x, orc.params_from_workload(wl), heads=[(0, 3), (1, 12)])
    compare(g32, ref, label="c3c", fp32_out=True)
    g = run_gpu(wl, x)
    compare(g, ref, label="c3c")
    check_bf16_is_rounded_fp32(g, g32, "c3c")
    assert torch.isfinite(g["O"]).all()


def test_causal_cuda_graph_capture_and_replay():
    """The causal forward (work counters reset, side-stream fork and join)
    captured into a CUDA graph and replayed on new inputs in the same
    buffers: bit-identical to an eager call, and to the oracle."""
    wl = small(H=2, N=1024, d_h=128, block=128, race_tables=16)
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl)
    x1 = make_inputs(wl)
    x2 = make_inputs(wl.with_(seed=wl.seed + 1))
    xd = {k: v.to(dev) for k, v in x1.items()}
    o = torch.empty_like(xd["q"])
    ws = elsaa.new_workspace(p, dev)
    st = torch.cuda.Stream(dev)

    def call():
        elsaa.elsaa_forward(p, xd["q"], xd["k"], xd["v"], xd["w_sort"],
                            xd["w_race"], o=o, workspace=ws, stream=st)

    with torch.cuda.stream(st):
        call()
    st.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=st):
        call()
    for k in xd:
        xd[k].copy_(x2[k].to(dev))
    o.zero_()
    graph.replay()
    graph.replay()  # counters are reset inside the graph
    torch.cuda.synchronize()
    elsaa.elsaa_check_status(ws)
    replay = o.clone()
    with torch.cuda.stream(st):
        call()
    st.synchronize()
    assert torch.equal(replay, o)
    ref = oc.forward(x2, orc.params_from_workload(wl))
    for (b, h), r in ref.items():
        assert o_err(replay[b, h].float().cpu().numpy(), r["O"]) <= 1.0
