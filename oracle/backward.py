"""Analytic gradient of the ELSAA operator for one head (fp64, numpy).

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: the tests, the
benchmark's CPU baseline and ``__graft_entry__.smoke()`` are the only
callers; nothing here is imported by the CUDA product path.

The paper trains ELSAA end to end but prints no backward pass; this module
differentiates the forward definitions it does print, in their order:

* sortLSH (Algorithm "sortLSH Sparse Exact Attention Branch"): per sorted
  block t, z_ij = scale <Q_i, K_j>, d_s,i = sum_j exp(z_ij),
  O_s,i = sum_j exp(z_ij) V_j / (d_s,i + eps). The hash and the sort are
  piecewise constant: they contribute no gradient, so the permutations of
  the forward pass are reused as given.
* RACE (Algorithm "RACE Low-Rank Attention Branch"): u = tanh(W^l x),
  phi^l(x)_r = softmax_r(beta u^T v_r) over the 2^gamma corners v_r of
  {-1, +1}^gamma, A^l = sum_j phi^l(K_j), B^l = sum_j phi^l(K_j) V_j^T,
  Num_i = (1/L) sum_l phi^l(Q_i)^T B^l, Den_i = (1/L) sum_l phi^l(Q_i).A^l,
  O_lr,i = Num_i / (Den_i + eps), d_lr,i = Den_i.
* Fusion, Eq. (5)-(6): D_i = d_s,i + lambda_i d_lr,i + eps,
  m_i = d_s,i / D_i (m_i = 1 in the Sort_LSH_RACE ablation),
  O_i = g_s,i m_i O_s,i + g_lr,i O_lr,i.

Every step is the chain rule written out on whole arrays; numpy's matmul is
the only library routine used. Corner labels: v_{r,b} = +1 if bit b of r is
set, else -1 (the forward oracle's labelling).
"""
from __future__ import annotations

import numpy as np


def corners(gamma: int) -> np.ndarray:
    """v[r, b] in {-1, +1}: +1 where bit b of r is set."""
    r = np.arange(1 << gamma)[:, None]
    b = np.arange(gamma)[None, :]
    return np.where((r >> b) & 1, 1.0, -1.0)


def race_phi(X: np.ndarray, W: np.ndarray, beta: float):
    """Soft hash of rows X[n, d] for planes W[L, gamma, d].

    Returns (phi[n, L, R], u[n, L, gamma]): u = tanh(W^l x), phi the softmax
    over corners of beta u^T v_r (Algorithm RACE, the feature step)."""
    L, gamma, _ = W.shape
    u = np.tanh(np.einsum("lgd,nd->nlg", W, X))
    a = beta * np.einsum("nlg,rg->nlr", u, corners(gamma))
    a = a - a.max(axis=2, keepdims=True)
    e = np.exp(a)
    return e / e.sum(axis=2, keepdims=True), u


def race_phi_grad(gphi, phi, u, W, beta):
    """dL/dx[n, d] from dL/dphi[n, L, R] through the softmax over corners,
    beta u^T v_r, u = tanh(W^l x)."""
    gamma = W.shape[1]
    ga = phi * (gphi - (phi * gphi).sum(axis=2, keepdims=True))
    gu = beta * np.einsum("nlr,rg->nlg", ga, corners(gamma))
    gwx = (1.0 - u * u) * gu
    return np.einsum("nlg,lgd->nd", gwx, W)


def forward_fixed_perm(Q, K, V, W, perm_q, perm_k, p, lam=None, gates=None):
    """The forward definitions above for given permutations, fp64, all rows
    (returns the pieces the gradient needs)."""
    N, d = Q.shape
    b = p["block"]
    scale = p["scale"] if p.get("scale") else 1.0 / np.sqrt(d)
    eps = p["eps"]
    # sortLSH: block t of sorted queries against block t of sorted keys
    O_s = np.zeros((N, d))
    d_s = np.zeros(N)
    for t in range(N // b):
        iq = perm_q[t * b:(t + 1) * b]
        ik = perm_k[t * b:(t + 1) * b]
        E = np.exp(scale * Q[iq] @ K[ik].T)
        d_s[iq] = E.sum(axis=1)
        O_s[iq] = (E @ V[ik]) / (d_s[iq] + eps)[:, None]
    # RACE
    L = W.shape[0]
    phi_k, _ = race_phi(K, W, p["beta"])
    phi_q, _ = race_phi(Q, W, p["beta"])
    A = phi_k.sum(axis=0)                             # [L, R]
    B = np.einsum("jlr,jd->lrd", phi_k, V)            # [L, R, d]
    Num = np.einsum("ilr,lrd->id", phi_q, B) / L
    Den = np.einsum("ilr,lr->i", phi_q, A) / L
    O_lr = Num / (Den + eps)[:, None]
    # fusion
    lam_v = np.full(N, p["lam"]) if lam is None else np.asarray(lam, np.float64)
    g_s = np.ones(N) if gates is None else np.asarray(gates, np.float64)[:, 0]
    g_lr = np.ones(N) if gates is None else np.asarray(gates, np.float64)[:, 1]
    D = d_s + lam_v * Den + eps
    m = d_s / D if p["fusion_mode"] == 0 else np.ones(N)
    O = (g_s * m)[:, None] * O_s + g_lr[:, None] * O_lr
    return dict(O=O, O_s=O_s, d_s=d_s, O_lr=O_lr, Den=Den, Num=Num, A=A,
                B=B, phi_q=phi_q, phi_k=phi_k, D=D, m=m, lam=lam_v, g_s=g_s,
                g_lr=g_lr, scale=scale)


def backward_fixed_perm(Q, K, V, W, perm_q, perm_k, G, p, lam=None,
                        gates=None):
    """Gradient of sum(G * O) w.r.t. Q, K, V, the gates and lambda (fp64)."""
    N, d = Q.shape
    b = p["block"]
    eps = p["eps"]
    beta = p["beta"]
    L = W.shape[0]
    f = forward_fixed_perm(Q, K, V, W, perm_q, perm_k, p, lam, gates)
    scale = f["scale"]
    d_s, D, m = f["d_s"], f["D"], f["m"]
    O_s, O_lr, Den = f["O_s"], f["O_lr"], f["Den"]
    g_s, g_lr, lam_v = f["g_s"], f["g_lr"], f["lam"]

    # Eq. (6): O = g_s m O_s + g_lr O_lr
    GO_s = np.einsum("id,id->i", G, O_s)
    dg_s = m * GO_s
    dg_lr = np.einsum("id,id->i", G, O_lr)
    dO_s = (g_s * m)[:, None] * G
    dO_lr = g_lr[:, None] * G
    # Eq. (5): m = d_s / D, D = d_s + lambda d_lr + eps
    if p["fusion_mode"] == 0:
        dm = g_s * GO_s
        dds_m = dm * (lam_v * Den + eps) / D ** 2
        dlr_m = -dm * lam_v * d_s / D ** 2
        dlam = -dm * d_s * Den / D ** 2
    else:
        dds_m = np.zeros(N)
        dlr_m = np.zeros(N)
        dlam = np.zeros(N)

    dQ = np.zeros((N, d))
    dK = np.zeros((N, d))
    dV = np.zeros((N, d))

    # sortLSH: O_s = Ns / (d_s + eps), Ns = sum_j exp(z) V_j, d_s = sum exp(z)
    gNs = dO_s / (d_s + eps)[:, None]
    gds = -np.einsum("id,id->i", dO_s, O_s) / (d_s + eps) + dds_m
    for t in range(N // b):
        iq = perm_q[t * b:(t + 1) * b]
        ik = perm_k[t * b:(t + 1) * b]
        E = np.exp(scale * Q[iq] @ K[ik].T)
        dZ = E * (gNs[iq] @ V[ik].T + gds[iq][:, None])
        dQ[iq] += scale * dZ @ K[ik]
        dK[ik] += scale * dZ.T @ Q[iq]
        dV[ik] += E.T @ gNs[iq]

    # RACE: O_lr = Num / (Den + eps), d_lr = Den
    phi_q, phi_k, A, B = f["phi_q"], f["phi_k"], f["A"], f["B"]
    gNum = dO_lr / (Den + eps)[:, None]
    gDen = -np.einsum("id,id->i", dO_lr, O_lr) / (Den + eps) + dlr_m
    # Num_i = (1/L) sum phi_q B, Den_i = (1/L) sum phi_q . A
    gphi_q = (np.einsum("lrd,id->ilr", B, gNum)
              + np.einsum("lr,i->ilr", A, gDen)) / L
    gB = np.einsum("ilr,id->lrd", phi_q, gNum) / L
    gA = np.einsum("ilr,i->lr", phi_q, gDen) / L
    # B = sum_j phi_k V_j^T, A = sum_j phi_k
    dV += np.einsum("jlr,lrd->jd", phi_k, gB)
    gphi_k = np.einsum("lrd,jd->jlr", gB, V) + gA[None]
    _, u_q = race_phi(Q, W, beta)
    _, u_k = race_phi(K, W, beta)
    dQ += race_phi_grad(gphi_q, phi_q, u_q, W, beta)
    dK += race_phi_grad(gphi_k, phi_k, u_k, W, beta)
    return dict(dQ=dQ, dK=dK, dV=dV, dgates=np.stack([dg_s, dg_lr], axis=1),
                dlam=dlam, O=f["O"])


def backward_head(q32, k32, v32, w_sort, w_race, G, p, lam=None,
                  gates=None):
    """Gradient for one head from exact input values: the permutations come
    from the forward oracle's hash and stable sort (the same discrete
    decisions as the forward pass)."""
    from . import oracle as fwd

    N, d = q32.shape
    ws = w_sort if p["sort_bits"] > 0 else np.zeros((0, d), np.float32)
    perm_q = fwd.stable_argsort(fwd.sort_keys(q32, ws, p["gray"])[0])
    perm_k = fwd.stable_argsort(fwd.sort_keys(k32, ws, p["gray"])[0])
    out = backward_fixed_perm(
        np.asarray(q32, np.float64), np.asarray(k32, np.float64),
        np.asarray(v32, np.float64), np.asarray(w_race, np.float64),
        perm_q, perm_k, np.asarray(G, np.float64), p, lam, gates)
    out["perm_q"] = perm_q
    out["perm_k"] = perm_k
    return out
