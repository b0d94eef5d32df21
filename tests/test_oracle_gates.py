"""Pins of the gate-MLP / lambda oracle (oracle/gates.py). CPU only.

* torch (float64) evaluates the same MLP with its own Linear, SiLU and
  sigmoid: an independent implementation of every step.
* Closed forms: W2 = 0 gives gates = sigmoid(b2) in every row; W1 = 0 gives
  the constant hidden layer SiLU(b1); printed values of SiLU and sigmoid.
* lambda: w = 0 gives c + sigmoid(b); the lambda_min floor; the range
  [max(c, lambda_min), c + 1].
* Planted mistakes in a copy of gates.py each fail one of the pins.
"""
import importlib.util

import numpy as np
import pytest

from oracle import gates as og


def _case(N=40, d=16, g=8, seed=0):
    rng = np.random.default_rng(seed)
    return dict(Q=rng.standard_normal((N, d)) * 1.5,
                w1=rng.standard_normal((g, d)) / np.sqrt(d),
                b1=rng.standard_normal(g) * 0.3,
                w2=rng.standard_normal((2, g)) / np.sqrt(g),
                b2=rng.standard_normal(2) * 0.5,
                w=rng.standard_normal(d) * 0.2, b=0.1, c=0.3)


def check_pins(mod):
    torch = pytest.importorskip("torch")
    F = torch.nn.functional
    c = _case()
    # (1) torch float64: Linear -> SiLU -> Linear -> sigmoid
    t = lambda a: torch.tensor(np.asarray(a), dtype=torch.float64)
    ref = torch.sigmoid(F.linear(F.silu(F.linear(t(c["Q"]), t(c["w1"]),
                                                 t(c["b1"]))),
                                 t(c["w2"]), t(c["b2"]))).numpy()
    got = mod.gate_mlp_head(c["Q"], c["w1"], c["b1"], c["w2"], c["b2"])
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-13)
    ref_l = (c["c"] + torch.sigmoid(t(c["Q"]) @ t(c["w"]) + c["b"])).numpy()
    got_l = mod.lambda_head(c["Q"], c["w"], c["b"], c["c"], 1e-6)
    np.testing.assert_allclose(got_l, ref_l, rtol=0, atol=1e-13)

    # (2) W2 = 0: gates = sigmoid(b2) = (1/2, 3/4) for b2 = (0, ln 3)
    g = mod.gate_mlp_head(c["Q"], c["w1"], c["b1"], np.zeros((2, 8)),
                          np.array([0.0, np.log(3.0)]))
    np.testing.assert_allclose(g, np.tile([0.5, 0.75], (40, 1)), atol=1e-15)

    # (3) W1 = 0: hidden = SiLU(b1); b1 = (1, -1), W2 = I, b2 = 0
    g = mod.gate_mlp_head(c["Q"][:, :4], np.zeros((2, 4)),
                          np.array([1.0, -1.0]), np.eye(2), np.zeros(2))
    z = np.array([0.7310585786300049, -0.2689414213699951])
    np.testing.assert_allclose(g, np.tile(1 / (1 + np.exp(-z)), (40, 1)),
                               atol=1e-15)

    # (4) printed values and tails (no overflow)
    with np.errstate(over="raise"):
        s = mod.silu(np.array([0.0, 1.0, -1.0, 40.0, -800.0]))
        sg = mod.sigmoid(np.array([-800.0, 800.0, 0.0]))
    np.testing.assert_allclose(
        s[:3], [0.0, 0.7310585786300049, -0.2689414213699951], atol=1e-15)
    assert abs(s[3] - 40.0) < 1e-12 and s[4] == 0.0
    np.testing.assert_array_equal(sg, [0.0, 1.0, 0.5])
    x = np.linspace(-30, 30, 61)
    np.testing.assert_allclose(mod.sigmoid(x) + mod.sigmoid(-x), 1.0,
                               atol=1e-15)

    # (5) lambda: w = 0 -> c + sigmoid(b); floor; range
    lam = mod.lambda_head(c["Q"], np.zeros(16), 0.0, 0.3, 1e-6)
    np.testing.assert_allclose(lam, 0.8, atol=1e-15)
    lam = mod.lambda_head(c["Q"][:1] * 0 + 1.0, np.full(16, -100.0), 0.0,
                          0.0, 1e-6)
    assert lam[0] == 1e-6
    lam = mod.lambda_head(c["Q"], c["w"] * 20, -1.0, 0.25, 1e-6)
    assert lam.min() >= 0.25 and lam.max() <= 1.25
    assert lam.max() - lam.min() > 0.1


def test_oracle_gates_pins():
    check_pins(og)


def test_gates_lambda_batched_matches_per_head():
    rng = np.random.default_rng(4)
    B, H, N, d, g = 2, 3, 20, 8, 16
    Q = rng.standard_normal((B, H, N, d))
    mlp = dict(w1=rng.standard_normal((H, g, d)), b1=rng.standard_normal((H, g)),
               w2=rng.standard_normal((H, 2, g)), b2=rng.standard_normal((H, 2)),
               w_lambda=rng.standard_normal((H, d)), b_lambda=np.zeros(H),
               c_lambda=np.full(H, 0.3), lambda_min=1e-6)
    G, L = og.gates_lambda(Q, mlp)
    for b in range(B):
        for h in range(H):
            np.testing.assert_array_equal(
                G[b, h], og.gate_mlp_head(Q[b, h], mlp["w1"][h], mlp["b1"][h],
                                          mlp["w2"][h], mlp["b2"][h]))
            np.testing.assert_array_equal(
                L[b, h], og.lambda_head(Q[b, h], mlp["w_lambda"][h], 0.0, 0.3,
                                        1e-6))
    assert np.all((G > 0) & (G < 1))
    G2, _ = og.gates_lambda(Q, mlp, heads=[(1, 2)])
    assert np.isnan(G2[0, 0]).all()
    np.testing.assert_array_equal(G2[1, 2], G[1, 2])


MUTATIONS = [
    ("silu_is_sigmoid", "return x * sigmoid(x)", "return sigmoid(x)"),
    ("hidden_bias_dropped",
     "hidden = Q @ np.asarray(w1, np.float64).T + np.asarray(b1, np.float64)",
     "hidden = Q @ np.asarray(w1, np.float64).T"),
    ("output_sigmoid_dropped", "    return sigmoid(z)\n", "    return z\n"),
    ("negative_tail_sign", "out[~pos] = e / (1.0 + e)",
     "out[~pos] = 1.0 / (1.0 + e)"),
    ("lambda_floor_is_ceiling",
     "return np.maximum(float(c) + sigmoid(t), float(lambda_min))",
     "return np.minimum(float(c) + sigmoid(t), float(lambda_min))"),
    ("lambda_offset_dropped",
     "return np.maximum(float(c) + sigmoid(t), float(lambda_min))",
     "return np.maximum(sigmoid(t), float(lambda_min))"),
    ("output_bias_dropped",
     "z = a @ np.asarray(w2, np.float64).T + np.asarray(b2, np.float64)",
     "z = a @ np.asarray(w2, np.float64).T"),
]


@pytest.mark.parametrize("name,old,new", MUTATIONS,
                         ids=[m[0] for m in MUTATIONS])
def test_planted_gate_mistake_is_caught(tmp_path, name, old, new):
    src = open(og.__file__).read()
    assert src.count(old) == 1, name
    path = tmp_path / "mutant_gates.py"
    path.write_text(src.replace(old, new))
    spec = importlib.util.spec_from_file_location("mutant_gates", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    with pytest.raises(AssertionError):
        check_pins(mod)
