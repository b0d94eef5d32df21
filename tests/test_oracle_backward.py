"""Pins of the oracle's analytic gradient (oracle/backward.py). CPU only.

* Central finite differences of sum(G * O), with O from the C oracle's own
  forward pieces (independent code) at fixed permutations: every input
  coordinate checked here, plus the gates and the per-token lambda.
* One block, g = (1, 0), lambda = 0, eps = 0: the operator is dense softmax
  attention, and the gradient equals torch autograd through torch.softmax.
* beta = 0, g = (0, 1): phi is constant, O_lr = (1/R) sum_j V_j / (N/R + eps)
  in every row, so dV_j = sum_i G_i (1/R) / (N/R + eps) and dQ = dK = 0.
* Planted mistakes in a copy of backward.py each fail the finite-difference
  pin.
"""
import importlib.util

import numpy as np
import pytest

from oracle import oracle as orc
from oracle import backward as bwd


def make_case(N=96, d=16, b=32, L=2, gamma=3, n_s=3, seed=0, beta=1.0,
              eps=1e-3, lam_scale=1.0, mode=0):
    rng = np.random.default_rng(seed)
    q = (rng.standard_normal((N, d)) * 0.7).astype(np.float32)
    k = (rng.standard_normal((N, d)) * 0.7).astype(np.float32)
    v = rng.standard_normal((N, d)).astype(np.float32)
    w_sort = rng.standard_normal((n_s, d)).astype(np.float32)
    W = rng.standard_normal((L, gamma, d)) * 0.4
    G = rng.standard_normal((N, d))
    lam = np.abs(rng.standard_normal(N)) * lam_scale + 0.1
    gates = rng.uniform(0.2, 1.2, (N, 2))
    p = orc.default_params(block=b, sort_bits=n_s, beta=beta, eps=eps,
                           lam=1.0, fusion_mode=mode)
    perm_q = orc.stable_argsort(orc.sort_keys(q, w_sort, 1)[0])
    perm_k = orc.stable_argsort(orc.sort_keys(k, w_sort, 1)[0])
    return dict(Q=q.astype(np.float64), K=k.astype(np.float64),
                V=v.astype(np.float64), W=W, G=G, lam=lam, gates=gates, p=p,
                perm_q=perm_q, perm_k=perm_k)


def c_forward(Q, K, V, W, perm_q, perm_k, p, lam, gates):
    """O of all rows from the C oracle's pieces (fixed permutations)."""
    N, d = Q.shape
    rows = np.arange(N, dtype=np.int32)
    scale = p["scale"] if p.get("scale") else 1.0 / np.sqrt(d)
    O_s, d_s, log_d_s = orc.sortlsh_rows(Q, K, V, perm_q, perm_k, p["block"],
                                         scale, p["eps"], rows)
    A, Bs = orc.race_summaries(K, V, W, p["beta"])
    O_lr, d_lr = orc.race_readout_rows(Q, W, p["beta"], p["eps"], A, Bs, rows)
    O, _, _ = orc.fuse_rows(O_s, d_s, log_d_s, O_lr, d_lr, lam, gates[:, 0],
                            gates[:, 1], p["eps"], p["fusion_mode"])
    return O


def fd_check(c, backward_fn, n_coords=12, h=1e-5, seed=1, rtol=2e-5):
    g = backward_fn(c["Q"], c["K"], c["V"], c["W"], c["perm_q"], c["perm_k"],
                    c["G"], c["p"], c["lam"], c["gates"])
    rng = np.random.default_rng(seed)
    args = dict(Q=c["Q"], K=c["K"], V=c["V"], lam=c["lam"],
                gates=c["gates"])

    def loss(**over):
        a = dict(args)
        a.update(over)
        O = c_forward(a["Q"], a["K"], a["V"], c["W"], c["perm_q"],
                      c["perm_k"], c["p"], a["lam"], a["gates"])
        return float((c["G"] * O).sum())

    worst = 0.0
    for name, grad in (("Q", g["dQ"]), ("K", g["dK"]), ("V", g["dV"]),
                       ("gates", g["dgates"]), ("lam", g["dlam"])):
        x = args[name]
        for _ in range(n_coords):
            idx = tuple(rng.integers(0, s) for s in x.shape)
            xp = x.copy()
            xm = x.copy()
            xp[idx] += h
            xm[idx] -= h
            num = (loss(**{name: xp}) - loss(**{name: xm})) / (2 * h)
            ana = grad[idx]
            err = abs(num - ana) / max(1.0, abs(num))
            worst = max(worst, err)
            assert err < rtol, (name, idx, num, ana)
    return worst


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("gamma,L", [(3, 2), (4, 1)])
def test_gradient_matches_central_differences(mode, gamma, L):
    c = make_case(gamma=gamma, L=L, mode=mode, seed=gamma + 10 * mode)
    fd_check(c, bwd.backward_fixed_perm)


def test_gradient_small_eps_and_blocks_of_16():
    c = make_case(N=64, b=16, eps=1e-6, seed=7)
    fd_check(c, bwd.backward_fixed_perm)


def test_one_block_is_dense_attention_gradient():
    torch = pytest.importorskip("torch")
    N, d = 48, 8
    c = make_case(N=N, d=d, b=N, eps=0.0, seed=3)
    c["p"]["lam"] = 0.0
    gates = np.stack([np.ones(N), np.zeros(N)], axis=1)
    g = bwd.backward_fixed_perm(c["Q"], c["K"], c["V"], c["W"], c["perm_q"],
                                c["perm_k"], c["G"], c["p"], np.zeros(N),
                                gates)
    Qt = torch.tensor(c["Q"], requires_grad=True)
    Kt = torch.tensor(c["K"], requires_grad=True)
    Vt = torch.tensor(c["V"], requires_grad=True)
    O = torch.softmax(Qt @ Kt.T / np.sqrt(d), dim=1) @ Vt
    (O * torch.tensor(c["G"])).sum().backward()
    np.testing.assert_allclose(g["O"], O.detach().numpy(), atol=1e-12)
    for ours, ref in ((g["dQ"], Qt.grad), (g["dK"], Kt.grad),
                      (g["dV"], Vt.grad)):
        np.testing.assert_allclose(ours, ref.numpy(), atol=1e-10)


def test_beta_zero_race_gradient_closed_form():
    N, d, L, gamma, eps = 64, 8, 2, 3, 1e-3
    c = make_case(N=N, d=d, L=L, gamma=gamma, beta=0.0, eps=eps, seed=5)
    R = 1 << gamma
    gates = np.stack([np.zeros(N), np.ones(N)], axis=1)
    g = bwd.backward_fixed_perm(c["Q"], c["K"], c["V"], c["W"], c["perm_q"],
                                c["perm_k"], c["G"], c["p"], c["lam"], gates)
    want_dv = np.tile(c["G"].sum(axis=0) / R / (N / R + eps), (N, 1))
    np.testing.assert_allclose(g["dV"], want_dv, atol=1e-12)
    assert np.abs(g["dQ"]).max() < 1e-12
    assert np.abs(g["dK"]).max() < 1e-12


MUTATIONS = [
    ("softmax_backward_sign",
     "ga = phi * (gphi - (phi * gphi).sum(axis=2, keepdims=True))",
     "ga = phi * (gphi + (phi * gphi).sum(axis=2, keepdims=True))"),
    ("tanh_derivative_dropped", "gwx = (1.0 - u * u) * gu", "gwx = gu"),
    ("sparse_dv_transposed", "dV[ik] += E.T @ gNs[iq]",
     "dV[ik] += E @ gNs[iq]"),
    ("multiplier_term_dropped",
     "gds = -np.einsum(\"id,id->i\", dO_s, O_s) / (d_s + eps) + dds_m",
     "gds = -np.einsum(\"id,id->i\", dO_s, O_s) / (d_s + eps)"),
    ("table_average_dropped_in_gB",
     "gB = np.einsum(\"ilr,id->lrd\", phi_q, gNum) / L",
     "gB = np.einsum(\"ilr,id->lrd\", phi_q, gNum)"),
    ("den_gradient_sign",
     "gDen = -np.einsum(\"id,id->i\", dO_lr, O_lr) / (Den + eps) + dlr_m",
     "gDen = np.einsum(\"id,id->i\", dO_lr, O_lr) / (Den + eps) + dlr_m"),
    ("key_scale_dropped", "dK[ik] += scale * dZ.T @ Q[iq]",
     "dK[ik] += dZ.T @ Q[iq]"),
]


@pytest.mark.parametrize("name,old,new", MUTATIONS,
                         ids=[m[0] for m in MUTATIONS])
def test_planted_gradient_mistake_is_caught(tmp_path, name, old, new):
    src = open(bwd.__file__).read()
    assert src.count(old) == 1, name
    path = tmp_path / "mutant_backward.py"
    path.write_text(src.replace(old, new))
    spec = importlib.util.spec_from_file_location("mutant_backward", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    c = make_case(seed=11)
    with pytest.raises(AssertionError):
        fd_check(c, mod.backward_fixed_perm)
