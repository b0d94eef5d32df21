"""Causal ELSAA oracle (numpy fp64): Algorithm "Causal RACE Low-Rank
Attention Branch", Algorithm "Causal sortLSH Sparse Exact Attention Branch"
(CausalSparse, SortLSH, MergeLSE) and Algorithm "Causal ELSAA" (the
log-domain multiplier of Eq. (5) and the fusion of Eq. (6)).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's ``cpu_baseline`` / ``--impl reference`` leg are the only callers.
The CUDA product path never imports this module, and this module imports
nothing from the product package.

Each function follows the algorithm's steps in the paper's order. Readings
where the paper is silent:

* CR1 the exact causal attention of a base segment uses the same epsilon
  placement as the non-causal sparse branch: O_i = sum_{j<=i} e^{z_ij} V_j /
  (d_i + eps), log d_i = log sum_{j<=i} e^{z_ij};
* CR2 a padding token (odd n) is a zero vector for Q, K and V; it is hashed
  like any other row (all projections 0, so every sign bit is 0);
* CR3 the SortLSH call on (Q_f, K_p, V_p) uses the same planes and code
  order as the non-causal branch; when m is not a multiple of b the last
  sorted block is shorter (the same length on both sides, since both halves
  hold m rows);
* CR4 in Causal RACE the padded positions carry zero features (they come
  after every real key and are masked for every real query, so their value
  does not reach any output);
* CR5 the fusion takes d_s = exp(log d_s) of the merged sparse result.
"""
from __future__ import annotations

import numpy as np

from . import oracle as orc


# ------------------------------------------------------------ sparse branch

def exact_causal(Q, K, V, scale, eps):
    """Exact causal attention of one segment (CR1): rows i attend keys
    j <= i of the same segment. Returns (O [n, d], log d [n])."""
    n = Q.shape[0]
    z = scale * (Q @ K.T)
    z[np.triu_indices(n, 1)] = -np.inf
    zmax = z.max(axis=1, keepdims=True)
    e = np.exp(z - zmax)
    s = e.sum(axis=1)
    logd = zmax[:, 0] + np.log(s)
    # sum e^z V / (sum e^z + eps), evaluated with the row maximum factored out
    O = (e @ V) / (s + eps * np.exp(-zmax[:, 0]))[:, None]
    return O, logd


def sortlsh_pair(Q, K, V, hq, hk, b, scale, eps, orders=None):
    """Algorithm sortLSH on queries Q and keys K, V of the same length m
    with codes hq, hk: stable sort of both, blocks of b consecutive sorted
    positions (the last one shorter if b does not divide m, CR3), query
    block t attends key block t. Returns (O, log d) in the original query
    order. When `orders` is a list, the two sorted orders (pq, pk; sorted
    position -> local row) are appended to it: they fix which keys each
    query attends."""
    m = Q.shape[0]
    pq = orc.stable_argsort(hq)
    pk = orc.stable_argsort(hk)
    if orders is not None:
        orders.append((pq, pk))
    O = np.zeros_like(Q)
    logd = np.zeros(m)
    for t0 in range(0, m, b):
        qi = pq[t0:t0 + b]
        kj = pk[t0:t0 + b]
        z = scale * (Q[qi] @ K[kj].T)
        zmax = z.max(axis=1, keepdims=True)
        e = np.exp(z - zmax)
        s = e.sum(axis=1)
        logd[qi] = zmax[:, 0] + np.log(s)
        O[qi] = (e @ V[kj]) / (s + eps * np.exp(-zmax[:, 0]))[:, None]
    return O, logd


def merge_lse(O1, ld1, O2, ld2, eps):
    """MergeLSE: mu = max(log d_1, log d_2), w_k = exp(log d_k - mu),
    s = w_1 + w_2, O = (w_1 O_1 + w_2 O_2) / (s + eps),
    log d = mu + log(s + eps)."""
    mu = np.maximum(ld1, ld2)
    w1 = np.exp(ld1 - mu)
    w2 = np.exp(ld2 - mu)
    s = w1 + w2
    O = (w1[:, None] * O1 + w2[:, None] * O2) / (s + eps)[:, None]
    return O, mu + np.log(s + eps)


def causal_sparse(Q, K, V, hq, hk, pad_code, b, N0, scale, eps, trace=None,
                  _start=0, _level=1):
    """CausalSparse(Q, K, V): the recursion of Algorithm "Causal sortLSH"
    over rows [0, n). hq, hk: sort codes of the rows; pad_code: the code of
    a zero row (CR2). Returns (O [n, d], log d [n]). When `trace` is a
    list, every SortLSH call of the recursion appends (level, first row of
    its node, sorted future-half query rows, sorted past-half key rows),
    rows counted from the start of the sequence, level 1 = the top."""
    n, d = Q.shape
    if n <= N0:
        return exact_causal(Q, K, V, scale, eps)
    padded = n % 2 == 1
    if padded:  # one zero token at the end, removed on return
        z = np.zeros((1, d))
        Q, K, V = (np.vstack([a, z]) for a in (Q, K, V))
        hq = np.append(hq, pad_code).astype(hq.dtype)
        hk = np.append(hk, pad_code).astype(hk.dtype)
        n += 1
    m = n // 2
    O_top, ld_top = causal_sparse(Q[:m], K[:m], V[:m], hq[:m], hk[:m],
                                  pad_code, b, N0, scale, eps, trace,
                                  _start, _level + 1)
    O_diag, ld_diag = causal_sparse(Q[m:], K[m:], V[m:], hq[m:], hk[m:],
                                    pad_code, b, N0, scale, eps, trace,
                                    _start + m, _level + 1)
    orders = [] if trace is not None else None
    O_off, ld_off = sortlsh_pair(Q[m:], K[:m], V[:m], hq[m:], hk[:m], b,
                                 scale, eps, orders)
    if trace is not None:
        pq, pk = orders[0]
        trace.append((_level, _start, _start + m + pq, _start + pk))
    O_bot, ld_bot = merge_lse(O_diag, ld_diag, O_off, ld_off, eps)
    O = np.vstack([O_top, O_bot])
    ld = np.concatenate([ld_top, ld_bot])
    if padded:
        O, ld = O[:-1], ld[:-1]
    return O, ld


# -------------------------------------------------------------- RACE branch

def race_features_rows(X, w_race, beta):
    """Phi^(l)(x) of every row of X: [n, L, R] (Algorithm RACE steps 3-7,
    through the C oracle's per-vector features)."""
    w = np.asarray(w_race, np.float64)
    L, gamma, _ = w.shape
    out = np.zeros((X.shape[0], L, 1 << gamma))
    for i in range(X.shape[0]):
        out[i] = orc.race_features(X[i], w, beta)
    return out


def causal_race(Q, K, V, w_race, beta, C, eps, phiQ=None, phiK=None):
    """Algorithm "Causal RACE Low-Rank Attention Branch". Returns
    (O_lr [N, d], d_lr [N])."""
    N, d = Q.shape
    L = np.asarray(w_race).shape[0]
    # soft hash features of every query and key, [N, L, R]
    if phiQ is None:
        phiQ = race_features_rows(Q, w_race, beta)
    if phiK is None:
        phiK = race_features_rows(K, w_race, beta)
    R = phiQ.shape[2]
    # pad the sequence axis to N' = ceil(N / C) C and cut it into chunks (CR4)
    n_c = -(-N // C)
    Np = n_c * C
    pQ = np.zeros((Np, L, R))
    pK = np.zeros((Np, L, R))
    pV = np.zeros((Np, d))
    pQ[:N], pK[:N], pV[:N] = phiQ, phiK, V
    # per table and chunk: A_n = Phi_K,n^T 1, B_n = Phi_K,n^T V_n
    A = np.zeros((n_c, L, R))
    B = np.zeros((n_c, L, R, d))
    for c in range(n_c):
        sl = slice(c * C, (c + 1) * C)
        for l in range(L):
            A[c, l] = pK[sl, l].sum(axis=0)
            B[c, l] = pK[sl, l].T @ pV[sl]
    # strict prefix states: cumulative sum, shifted right by one chunk
    sA = np.zeros_like(A)
    sB = np.zeros_like(B)
    sA[1:] = np.cumsum(A, axis=0)[:-1]
    sB[1:] = np.cumsum(B, axis=0)[:-1]
    tril = np.tril(np.ones((C, C)))
    O = np.zeros((Np, d))
    dlr = np.zeros(Np)
    for c in range(n_c):
        sl = slice(c * C, (c + 1) * C)
        # inter-chunk: queries read every earlier chunk's keys
        inum = sum(pQ[sl, l] @ sB[c, l] for l in range(L)) / L
        iden = sum(pQ[sl, l] @ sA[c, l] for l in range(L)) / L
        # intra-chunk: causally masked soft attention within the chunk
        Mn = sum(pQ[sl, l] @ pK[sl, l].T for l in range(L)) / L * tril
        anum = Mn @ pV[sl]
        aden = Mn.sum(axis=1)
        dlr[sl] = iden + aden
        O[sl] = (inum + anum) / (dlr[sl] + eps)[:, None]
    return O[:N], dlr[:N]


# ------------------------------------------------------------ whole operator

def forward_head(q32, k32, v32, w_sort, w_race, p: dict, lam=None,
                 gates=None) -> dict:
    """Algorithm "Causal ELSAA" for one head (after the projections).
    p: oracle params plus causal_chunk (C) and causal_base_len (N0)."""
    N, d = q32.shape
    scale = p["scale"] if p.get("scale") else 1.0 / np.sqrt(d)
    ws = w_sort if p["sort_bits"] > 0 else np.zeros((0, d), np.float32)
    hq, _ = orc.sort_keys(q32, ws, p["gray"])
    hk, _ = orc.sort_keys(k32, ws, p["gray"])
    pad_code = orc.sort_keys(np.zeros((1, d), np.float32), ws, p["gray"])[0][0]
    Q = q32.astype(np.float64)
    K = k32.astype(np.float64)
    V = v32.astype(np.float64)
    O_lr, d_lr = causal_race(Q, K, V, w_race, p["beta"], p["causal_chunk"],
                             p["eps"])
    trace = []
    O_s, log_d_s = causal_sparse(Q, K, V, hq, hk, pad_code, p["block"],
                                 p["causal_base_len"], scale, p["eps"],
                                 trace)
    lam_r = (np.full(N, p["lam"], np.float64) if lam is None
             else np.asarray(lam, np.float64))
    if gates is None:
        g_s = np.ones(N)
        g_lr = np.ones(N)
    else:
        g = np.asarray(gates, np.float64)
        g_s, g_lr = g[:, 0], g[:, 1]
    # log D = LSE(log d_s, log lambda + log d_lr, log eps); m = exp(log d_s -
    # log D); O = g_s m O_s + g_lr O_lr (CR5)
    O, m, m_log = orc.fuse_rows(O_s, np.exp(log_d_s), log_d_s, O_lr, d_lr,
                                lam_r, g_s, g_lr, p["eps"], p["fusion_mode"])
    return dict(O=O, O_sparse=O_s, log_d_sparse=log_d_s, O_lr=O_lr,
                d_lr=d_lr, m=m, m_log=m_log, keys_q=hq, keys_k=hk,
                index_lists=index_lists(trace))


def index_lists(trace):
    """The SortLSH orders of a trace of causal_sparse as per-level arrays:
    {level: (queries, keys)}, each the concatenation over the level's nodes
    (in row order) of the sorted row indices of the node's future-half
    queries and past-half keys."""
    out = {}
    for level in sorted({t[0] for t in trace}):
        nodes = sorted((t for t in trace if t[0] == level),
                       key=lambda t: t[1])
        out[level] = (np.concatenate([t[2] for t in nodes]),
                      np.concatenate([t[3] for t in nodes]))
    return out


def forward(inputs: dict, p: dict, lam=None, gates=None, heads=None) -> dict:
    """Causal ELSAA over [B, H, N, d_h] inputs for the listed (b, h) heads
    (None = all). Returns {(b, h): forward_head result}."""
    q = orc.to_numpy32(inputs["q"])
    k = orc.to_numpy32(inputs["k"])
    v = orc.to_numpy32(inputs["v"])
    w_sort = orc.to_numpy32(inputs["w_sort"])
    w_race = orc.to_numpy32(inputs["w_race"]).astype(np.float64)
    lam_a = None if lam is None else orc.to_numpy32(lam)
    gates_a = None if gates is None else orc.to_numpy32(gates)
    if heads is None:
        heads = [(b, h) for b in range(q.shape[0]) for h in range(q.shape[1])]
    return {(b, h): forward_head(
        q[b, h], k[b, h], v[b, h], w_sort[h], w_race[h], p,
        lam=None if lam_a is None else lam_a[b, h],
        gates=None if gates_a is None else gates_a[b, h])
        for b, h in heads}
