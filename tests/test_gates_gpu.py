"""GPU gate MLP and query-dependent lambda (elsaa_gates through the C ABI)
versus the fp64 oracle (oracle/gates.py) on the same seeded inputs.

Tolerance: the tensor-core path multiplies bf16 Q by bf16-representable W1
exactly and accumulates in fp32 (d_h <= 128 terms), then applies SiLU,
the 2 x g output layer and the sigmoids in fp32: the gates and lambda stay
within about 1e-5 of the fp64 values; the bound written here is 1e-4
absolute (gates lie in (0, 1), lambda in [c, c + 1]).
"""
import numpy as np
import pytest
import torch

from oracle import gates as og
from oracle import oracle as orc
from paper_2607_20214_gb300 import build, elsaa
from paper_2607_20214_gb300.workloads import (WORKLOADS, Workload,
                                              make_gate_mlp, make_inputs)

pytestmark = pytest.mark.gpu

TOL = 1e-4


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    elsaa.load_library()


def small(dtype="bf16", **kw):
    base = dict(name="gates", B=2, H=3, N=1184, d_h=128, dtype=dtype,
                block=32, race_tables=4, recipe="plain", temperature=2.0,
                seed=31, plane_seed=1031)
    base.update(kw)
    return Workload(**base)


def run_gates(wl, x, mlp):
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl)
    md = {k: (v.to(dev) if isinstance(v, torch.Tensor) else v)
          for k, v in mlp.items()}
    g, lam = elsaa.elsaa_gates(p, md, x["q"].to(dev))
    torch.cuda.synchronize()
    return g.cpu(), (None if lam is None else lam.cpu())


def oracle_gates(x, mlp, heads=None):
    npm = {k: (v.double().numpy() if isinstance(v, torch.Tensor) else v)
           for k, v in mlp.items()}
    return og.gates_lambda(x["q"].double().numpy(), npm, heads=heads)


@pytest.mark.parametrize("dtype,d_h,hidden", [
    ("bf16", 128, 64), ("bf16", 64, 128), ("bf16", 64, 16),
    ("bf16", 128, 128), ("fp32", 64, 64), ("bf16", 32, 32),
    ("fp32", 128, 16)])
def test_gates_match_oracle(dtype, d_h, hidden):
    wl = small(dtype, d_h=d_h)
    x = make_inputs(wl)
    mlp = make_gate_mlp(wl, hidden=hidden, seed=hidden + d_h)
    g, lam = run_gates(wl, x, mlp)
    rg, rl = oracle_gates(x, mlp)
    assert np.isfinite(g.numpy()).all() and np.isfinite(lam.numpy()).all()
    np.testing.assert_allclose(g.numpy(), rg, rtol=0, atol=TOL)
    np.testing.assert_allclose(lam.numpy(), rl, rtol=0, atol=TOL)
    # the inputs make both outputs vary (a constant would pass trivially)
    assert rg.std() > 0.05 and rl.std() > 0.01


def test_gates_without_lambda_and_floor():
    wl = small("bf16", d_h=64, B=1, H=2, N=512)
    x = make_inputs(wl)
    mlp = make_gate_mlp(wl, hidden=32, seed=5)
    no_l = dict(mlp, w_lambda=None)
    g, lam = run_gates(wl, x, no_l)
    assert lam is None
    rg, _ = oracle_gates(x, no_l)
    np.testing.assert_allclose(g.numpy(), rg, rtol=0, atol=TOL)
    # c = 0 and a strongly negative projection: lambda sits on the floor
    floor = dict(mlp, c_lambda=torch.zeros(wl.H),
                 b_lambda=torch.full((wl.H,), -200.0))
    _, lam = run_gates(wl, x, floor)
    assert (lam.numpy() == np.float32(1e-6)).all()


def test_learned_gates_feed_the_forward_pass():
    """elsaa_gates then elsaa_forward on one stream equals the oracle's
    fusion with the oracle's gates and lambda (Eq. (6))."""
    wl = small("bf16", d_h=64, block=64, B=1, H=2, N=1024)
    x = make_inputs(wl)
    mlp = make_gate_mlp(wl, hidden=64, seed=9)
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl)
    xd = {k: v.to(dev) for k, v in x.items()}
    md = {k: (v.to(dev) if isinstance(v, torch.Tensor) else v)
          for k, v in mlp.items()}
    g, lam = elsaa.elsaa_gates(p, md, xd["q"])
    o = elsaa.elsaa_forward(p, xd["q"], xd["k"], xd["v"], xd["w_sort"],
                            xd["w_race"], lambda_tok=lam, gates=g)
    torch.cuda.synchronize()
    rg, rl = oracle_gates(x, mlp)
    pr = orc.params_from_workload(wl)
    ref = orc.forward(x, pr, lam=rl, gates=rg, heads=[(0, 0), (0, 1)])
    for (b, h), r in ref.items():
        err = np.abs(o[b, h].float().cpu().numpy() - np.asarray(r["O"])).max()
        assert err <= 2e-2, (b, h, err)


def test_c3_full_size_gates():
    """All 524288 query rows of the N = 16384 workload (B = 2, H = 16,
    d_h = 128), hidden width 64 as in the paper's text setting."""
    wl = WORKLOADS["c3"]
    x = make_inputs(wl)
    mlp = make_gate_mlp(wl, hidden=64, seed=3)
    g, lam = run_gates(wl, x, mlp)
    rg, rl = oracle_gates(x, mlp)
    assert np.abs(g.numpy() - rg).max() <= TOL
    assert np.abs(lam.numpy() - rl).max() <= TOL


def run_gated(wl, x, mlp, **over):
    """elsaa_forward_gated: returns O, gates, lambda and the kernels that
    ran."""
    dev = torch.device("cuda:0")
    p = elsaa.params_for(wl, **over)
    xd = {k: v.to(dev) for k, v in x.items()}
    md = {k: (v.to(dev) if isinstance(v, torch.Tensor) else v)
          for k, v in mlp.items()}
    BHN = (wl.B, wl.H, wl.N)
    gts = torch.full(BHN + (2,), float("nan"), device=dev)
    lam = torch.full(BHN, float("nan"), device=dev) \
        if mlp.get("w_lambda") is not None else None
    elsaa.elsaa_profile_start()
    o = elsaa.elsaa_forward_gated(p, md, xd["q"], xd["k"], xd["v"],
                                  xd["w_sort"], xd["w_race"], gates_out=gts,
                                  lambda_out=lam)
    prof = elsaa.elsaa_profile_stop()
    torch.cuda.synchronize()
    return (o.float().cpu(), gts.cpu(), None if lam is None else lam.cpu(),
            prof)


@pytest.mark.parametrize("dtype,d_h,hidden,b", [
    ("bf16", 128, 64, 128), ("bf16", 64, 64, 64), ("bf16", 128, 16, 32),
    ("bf16", 64, 128, 128), ("bf16", 128, 48, 256), ("fp32", 64, 32, 32)])
def test_gated_forward_matches_oracle(dtype, d_h, hidden, b):
    """elsaa_forward_gated (the gate network inside the forward call):
    gates and lambda within 1e-4 of the oracle, O within the dtype's bound
    of the oracle's fusion with the oracle's gates."""
    wl = small(dtype, d_h=d_h, block=b, B=1, H=3, N=b * 10)
    x = make_inputs(wl)
    mlp = make_gate_mlp(wl, hidden=hidden, seed=hidden + d_h + 1)
    o, g, lam, prof = run_gated(wl, x, mlp)
    assert "gate_mlp" in prof and "sort_hash" in prof, prof
    rg, rl = oracle_gates(x, mlp)
    np.testing.assert_allclose(g.numpy(), rg, rtol=0, atol=TOL)
    np.testing.assert_allclose(lam.numpy(), rl, rtol=0, atol=TOL)
    ref = orc.forward(x, orc.params_from_workload(wl), lam=rl, gates=rg)
    bound = 2e-2 if dtype == "bf16" else 1e-4
    for (bb, h), r in ref.items():
        err = np.abs(o[bb, h].numpy() - np.asarray(r["O"])).max()
        assert err <= bound, (bb, h, err)


def test_gated_forward_equals_gates_then_forward():
    """The one call and elsaa_gates + elsaa_forward give the same gates and
    lambda; without lambda the scalar lambda is used; the causal variant
    takes the same gates."""
    wl = small("bf16", d_h=128, block=128, B=2, H=2, N=1280)
    x = make_inputs(wl)
    mlp = make_gate_mlp(wl, hidden=64, seed=77)
    o, g, lam, _ = run_gated(wl, x, mlp)
    g2, lam2 = run_gates(wl, x, mlp)
    assert torch.equal(g, g2) and torch.equal(lam, lam2)
    no_l = dict(mlp, w_lambda=None)
    o, g, lam, _ = run_gated(wl, x, no_l)
    assert lam is None
    rg, _ = oracle_gates(x, no_l)
    ref = orc.forward(x, orc.params_from_workload(wl), gates=rg,
                      heads=[(1, 1)])
    assert np.abs(o[1, 1].numpy() - ref[(1, 1)]["O"]).max() <= 2e-2
    wc = small("bf16", d_h=64, block=64, B=1, H=2, N=1024, causal=1,
               causal_base_len=256)
    xc = make_inputs(wc)
    mc = make_gate_mlp(wc, hidden=64, seed=79)
    o, g, lam, _ = run_gated(wc, xc, mc, out_fp32=1)
    rg, rl = oracle_gates(xc, mc)
    from oracle import causal as oc
    ref = oc.forward(xc, orc.params_from_workload(wc), lam=rl, gates=rg)
    for (bb, h), r in ref.items():
        assert np.abs(o[bb, h].numpy() - r["O"]).max() <= 2e-2


def test_c3_gated_forward_sampled():
    """c3 (B=2 H=16 N=16384 d_h=128, b=128, r=256) with hidden width 64:
    every gate and lambda, and O on sampled rows of two heads."""
    wl = WORKLOADS["c3"]
    x = make_inputs(wl)
    mlp = make_gate_mlp(wl, hidden=64, seed=3)
    o, g, lam, prof = run_gated(wl, x, mlp)
    assert "gate_mlp" in prof
    rg, rl = oracle_gates(x, mlp)
    assert np.abs(g.numpy() - rg).max() <= TOL
    assert np.abs(lam.numpy() - rl).max() <= TOL
    rows = np.sort(np.random.default_rng(8).choice(wl.N, 512, replace=False))
    ref = orc.forward(x, orc.params_from_workload(wl), lam=rl, gates=rg,
                      heads=[(0, 5), (1, 9)], rows=rows)
    for (bb, h), r in ref.items():
        err = np.abs(o[bb, h].numpy()[rows] - np.asarray(r["O"])).max()
        assert err <= 2e-2, (bb, h, err)
