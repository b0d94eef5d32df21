"""Token-wise gates and query-dependent lambda of the ELSAA fusion (fp64).

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: the tests, the
benchmark's CPU baseline and ``__graft_entry__.smoke()`` are the only
callers; nothing here is imported by the CUDA product path.

Definitions followed (per head, per query row q_i):

* Gates, Section 3.3 (the fusion paragraph) and Appendix D (model setup):
  (g_sparse,i, g_lr,i) = sigma(G_theta(q_i)), where G_theta is a two-layer
  MLP with a SiLU hidden activation and two outputs, each passed through
  its own sigmoid (no normalisation of the pair):
      a_i = SiLU(W1 q_i + b1)          (hidden width g)
      z_i = W2 a_i + b2                (2 outputs)
      g_i = sigmoid(z_i)               (elementwise)
  with SiLU(x) = x * sigmoid(x).
* Query-dependent lambda, Appendix D (the input-dependent version):
      lambda_i = max(c + sigmoid(w^T q_i + b), lambda_min),
  c >= 0, lambda_min = 1e-6 in the paper.

Every step is written out with numpy; nothing is fused or reordered.
"""
from __future__ import annotations

import numpy as np


def sigmoid(x):
    """1 / (1 + exp(-x)), evaluated without overflow on both tails."""
    x = np.asarray(x, np.float64)
    out = np.empty_like(x)
    pos = x >= 0
    out[pos] = 1.0 / (1.0 + np.exp(-x[pos]))
    e = np.exp(x[~pos])
    out[~pos] = e / (1.0 + e)
    return out


def silu(x):
    """SiLU(x) = x * sigmoid(x)."""
    x = np.asarray(x, np.float64)
    return x * sigmoid(x)


def gate_mlp_head(Q, w1, b1, w2, b2):
    """Gates [N, 2] of one head: sigmoid(W2 SiLU(W1 q + b1) + b2) per row.

    Q [N, d]; w1 [g, d]; b1 [g]; w2 [2, g]; b2 [2]."""
    Q = np.asarray(Q, np.float64)
    hidden = Q @ np.asarray(w1, np.float64).T + np.asarray(b1, np.float64)
    a = silu(hidden)
    z = a @ np.asarray(w2, np.float64).T + np.asarray(b2, np.float64)
    return sigmoid(z)


def lambda_head(Q, w, b, c, lambda_min):
    """lambda_i = max(c + sigmoid(w^T q_i + b), lambda_min) for one head."""
    Q = np.asarray(Q, np.float64)
    t = Q @ np.asarray(w, np.float64) + float(b)
    return np.maximum(float(c) + sigmoid(t), float(lambda_min))


def gates_lambda(Q, mlp: dict, heads=None):
    """Gates [B, H, N, 2] and lambda [B, H, N] (or None) for Q [B, H, N, d].

    ``mlp`` holds per-head arrays: w1 [H, g, d], b1 [H, g], w2 [H, 2, g],
    b2 [H, 2], and optionally w_lambda [H, d], b_lambda [H], c_lambda [H]
    with the scalar lambda_min. ``heads`` restricts the work to a list of
    (b, h) pairs (the other entries stay NaN)."""
    Q = np.asarray(Q, np.float64)
    B, H, N, _ = Q.shape
    gates = np.full((B, H, N, 2), np.nan)
    lam = None
    if mlp.get("w_lambda") is not None:
        lam = np.full((B, H, N), np.nan)
    todo = heads if heads is not None else [(b, h) for b in range(B)
                                            for h in range(H)]
    for (b, h) in todo:
        gates[b, h] = gate_mlp_head(Q[b, h], mlp["w1"][h], mlp["b1"][h],
                                    mlp["w2"][h], mlp["b2"][h])
        if lam is not None:
            lam[b, h] = lambda_head(Q[b, h], mlp["w_lambda"][h],
                                    mlp["b_lambda"][h], mlp["c_lambda"][h],
                                    mlp["lambda_min"])
    return gates, lam
