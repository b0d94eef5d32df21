"""Python front end of the ELSAA CPU oracle (fp64, plain C underneath).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's ``cpu_baseline`` / ``--impl reference`` leg are the only callers.
The CUDA product path never imports this module, and this module imports
nothing from the product package.

The C file ``elsaa_oracle.c`` implements the paper's steps for one head
(Algorithm sortLSH, Algorithm RACE, Eq. (5)-(6)); this wrapper loops over
heads (threads over heads: ctypes releases the GIL) and marshals arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "elsaa_oracle.c")
_LIB = os.path.join(_HERE, "libelsaa_oracle.so")

_dp = ctypes.POINTER(ctypes.c_double)
_fp = ctypes.POINTER(ctypes.c_float)
_ip = ctypes.POINTER(ctypes.c_int32)
_up = ctypes.POINTER(ctypes.c_uint16)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C, no fp contraction)."""
    if force or not os.path.exists(_LIB) or (
            os.path.getmtime(_LIB) < os.path.getmtime(_SRC)):
        tmp = _LIB + ".tmp%d" % os.getpid()
        subprocess.check_call([
            "gcc", "-O2", "-ffp-contract=off", "-fPIC", "-shared", "-std=c11",
            "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def configure(L):
    """Declare the C signatures on a loaded oracle library."""
    L.elsaa_oracle_sort_keys.restype = ctypes.c_int64
    L.elsaa_oracle_sort_keys.argtypes = [
        _fp, ctypes.c_int, ctypes.c_int, _fp, ctypes.c_int, ctypes.c_int,
        _up]
    L.elsaa_oracle_stable_argsort.argtypes = [_up, ctypes.c_int, _ip]
    L.elsaa_oracle_sortlsh.argtypes = [
        _dp, _dp, _dp, ctypes.c_int, ctypes.c_int, _ip, _ip, ctypes.c_int,
        ctypes.c_int, ctypes.c_double, ctypes.c_double, _dp, _dp, _dp]
    L.elsaa_oracle_sortlsh_rows.argtypes = [
        _dp, _dp, _dp, ctypes.c_int, ctypes.c_int, _ip, _ip, ctypes.c_int,
        ctypes.c_int, ctypes.c_double, ctypes.c_double, _ip, ctypes.c_int,
        _dp, _dp, _dp]
    L.elsaa_oracle_race_features.argtypes = [
        _dp, ctypes.c_int, _dp, ctypes.c_int, ctypes.c_int,
        ctypes.c_double, _dp]
    L.elsaa_oracle_race_summaries.argtypes = [
        _dp, _dp, ctypes.c_int, ctypes.c_int, _dp, ctypes.c_int,
        ctypes.c_int, ctypes.c_double, _dp, _dp]
    L.elsaa_oracle_race_readout_rows.argtypes = [
        _dp, ctypes.c_int, _dp, ctypes.c_int, ctypes.c_int,
        ctypes.c_double, ctypes.c_double, _dp, _dp, _ip, ctypes.c_int,
        _dp, _dp]
    L.elsaa_oracle_fuse_rows.argtypes = [
        ctypes.c_int, ctypes.c_int, _dp, _dp, _dp, _dp, _dp, _dp, _dp,
        _dp, ctypes.c_double, ctypes.c_int, _dp, _dp, _dp]
    L.elsaa_oracle_block_sums.argtypes = [
        _fp, ctypes.c_int, ctypes.c_int, _ip, ctypes.c_int, _fp]
    L.elsaa_oracle_topk_candidates.argtypes = [
        _fp, _fp, ctypes.c_int, ctypes.c_int, ctypes.c_int, _ip]
    L.elsaa_oracle_topk_select_rows.argtypes = [
        _fp, _fp, ctypes.c_int, ctypes.c_int, _ip, _ip, ctypes.c_int, _ip,
        ctypes.c_int, ctypes.c_int, _ip, ctypes.c_int, _ip]
    L.elsaa_oracle_sparse_sets_rows.argtypes = [
        _dp, _dp, _dp, ctypes.c_int, _ip, ctypes.c_int, ctypes.c_double,
        ctypes.c_double, _ip, ctypes.c_int, _dp, _dp, _dp]
    L.elsaa_oracle_dense_rows.argtypes = [
        _dp, _dp, _dp, ctypes.c_int, ctypes.c_int, ctypes.c_double, _ip,
        ctypes.c_int, _dp, _dp]
    return L


def lib():
    global _lib
    if _lib is None:
        _lib = configure(ctypes.CDLL(build()))
    return _lib


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _ptr(a, ct):
    return a.ctypes.data_as(ct)


def to_numpy32(t) -> np.ndarray:
    """Exact fp32 copy of a tensor/array (bf16 and fp32 widen exactly)."""
    if hasattr(t, "detach"):
        t = t.detach().to("cpu")
        import torch
        t = t.to(torch.float32).numpy()
    return _c(t, np.float32)


# ------------------------------------------------------------ single pieces

def sort_keys(x32: np.ndarray, w: np.ndarray, gray: int = 1):
    """Sort keys of rows x32[N, d_h]; returns (keys uint16[N], fp64 sign
    disagreements)."""
    x32 = _c(x32, np.float32)
    w = _c(w, np.float32)
    N, d = x32.shape
    n_s = w.shape[0] if w.ndim == 2 else 0
    keys = np.zeros(N, dtype=np.uint16)
    mism = lib().elsaa_oracle_sort_keys(
        _ptr(x32, _fp), N, d, _ptr(w if n_s else np.zeros((1, d), np.float32),
                                   _fp), n_s, gray, _ptr(keys, _up))
    return keys, int(mism)


def stable_argsort(keys: np.ndarray) -> np.ndarray:
    keys = _c(keys, np.uint16)
    perm = np.zeros(keys.shape[0], dtype=np.int32)
    lib().elsaa_oracle_stable_argsort(_ptr(keys, _up), keys.shape[0],
                                      _ptr(perm, _ip))
    return perm


def race_features(x: np.ndarray, w_race: np.ndarray, beta: float):
    """phi[L, R] of one vector x[d_h] for planes w_race[L, gamma, d_h]."""
    x = _c(x, np.float64)
    w = _c(w_race, np.float64)
    L, gamma, d = w.shape
    out = np.zeros((L, 1 << gamma), dtype=np.float64)
    lib().elsaa_oracle_race_features(_ptr(x, _dp), d, _ptr(w, _dp), L, gamma,
                                     beta, _ptr(out, _dp))
    return out


def race_summaries(K: np.ndarray, V: np.ndarray, w_race: np.ndarray,
                   beta: float):
    K = _c(K, np.float64)
    V = _c(V, np.float64)
    w = _c(w_race, np.float64)
    L, gamma, d = w.shape
    R = 1 << gamma
    A = np.zeros((L, R), dtype=np.float64)
    Bs = np.zeros((L, R, d), dtype=np.float64)
    lib().elsaa_oracle_race_summaries(_ptr(K, _dp), _ptr(V, _dp), K.shape[0],
                                      d, _ptr(w, _dp), L, gamma, beta,
                                      _ptr(A, _dp), _ptr(Bs, _dp))
    return A, Bs


def race_readout_rows(Q, w_race, beta, eps, A, Bs, rows):
    Q = _c(Q, np.float64)
    w = _c(w_race, np.float64)
    L, gamma, d = w.shape
    rows = _c(rows, np.int32)
    O = np.zeros((rows.shape[0], d), dtype=np.float64)
    dlr = np.zeros(rows.shape[0], dtype=np.float64)
    lib().elsaa_oracle_race_readout_rows(
        _ptr(Q, _dp), d, _ptr(w, _dp), L, gamma, beta, eps,
        _ptr(_c(A, np.float64), _dp), _ptr(_c(Bs, np.float64), _dp),
        _ptr(rows, _ip), rows.shape[0], _ptr(O, _dp), _ptr(dlr, _dp))
    return O, dlr


def sortlsh(Q, K, V, perm_q, perm_k, b, scale, eps, nb=0):
    """sortLSH branch of one head; query block t attends key blocks
    t - nb .. t + nb (clipped). Returns O_s, d_s, log d_s (all rows)."""
    Q = _c(Q, np.float64)
    K = _c(K, np.float64)
    V = _c(V, np.float64)
    N, d = Q.shape
    O = np.zeros((N, d), dtype=np.float64)
    ds = np.zeros(N, dtype=np.float64)
    lds = np.zeros(N, dtype=np.float64)
    lib().elsaa_oracle_sortlsh(
        _ptr(Q, _dp), _ptr(K, _dp), _ptr(V, _dp), N, d,
        _ptr(_c(perm_q, np.int32), _ip), _ptr(_c(perm_k, np.int32), _ip), b,
        nb, scale, eps, _ptr(O, _dp), _ptr(ds, _dp), _ptr(lds, _dp))
    return O, ds, lds


def sortlsh_rows(Q, K, V, perm_q, perm_k, b, scale, eps, rows, nb=0):
    Q = _c(Q, np.float64)
    K = _c(K, np.float64)
    V = _c(V, np.float64)
    N, d = Q.shape
    rows = _c(rows, np.int32)
    n = rows.shape[0]
    O = np.zeros((n, d), dtype=np.float64)
    ds = np.zeros(n, dtype=np.float64)
    lds = np.zeros(n, dtype=np.float64)
    lib().elsaa_oracle_sortlsh_rows(
        _ptr(Q, _dp), _ptr(K, _dp), _ptr(V, _dp), N, d,
        _ptr(_c(perm_q, np.int32), _ip), _ptr(_c(perm_k, np.int32), _ip), b,
        nb, scale, eps, _ptr(rows, _ip), n, _ptr(O, _dp), _ptr(ds, _dp),
        _ptr(lds, _dp))
    return O, ds, lds


def block_sums(x32, perm, b):
    """Top-k selector step 1: fp32 sums of each sorted block, [N / b, d]."""
    x32 = _c(x32, np.float32)
    N, d = x32.shape
    out = np.zeros((N // b, d), dtype=np.float32)
    lib().elsaa_oracle_block_sums(_ptr(x32, _fp), N, d,
                                  _ptr(_c(perm, np.int32), _ip), b,
                                  _ptr(out, _fp))
    return out


def topk_candidates(qsum, ksum, c):
    """Top-k selector step 2: candidate key blocks [T, c] of every query
    block (its own block first)."""
    qsum = _c(qsum, np.float32)
    ksum = _c(ksum, np.float32)
    T, d = qsum.shape
    cand = np.zeros((T, c), dtype=np.int32)
    lib().elsaa_oracle_topk_candidates(_ptr(qsum, _fp), _ptr(ksum, _fp), T,
                                       d, c, _ptr(cand, _ip))
    return cand


def topk_select_rows(q32, k32, perm_q, perm_k, b, cand, k, rows):
    """Top-k selector step 3: the k selected key indices of each of the
    query rows, [len(rows), k], increasing."""
    q32 = _c(q32, np.float32)
    k32 = _c(k32, np.float32)
    N, d = q32.shape
    cand = _c(cand, np.int32)
    rows = _c(rows, np.int32)
    sel = np.zeros((rows.shape[0], k), dtype=np.int32)
    lib().elsaa_oracle_topk_select_rows(
        _ptr(q32, _fp), _ptr(k32, _fp), N, d, _ptr(_c(perm_q, np.int32), _ip),
        _ptr(_c(perm_k, np.int32), _ip), b, _ptr(cand, _ip), cand.shape[1],
        k, _ptr(rows, _ip), rows.shape[0], _ptr(sel, _ip))
    return sel


def sparse_sets_rows(Q, K, V, sel, scale, eps, rows):
    """Top-k selector step 4: the sparse branch over each row's set."""
    Q = _c(Q, np.float64)
    K = _c(K, np.float64)
    V = _c(V, np.float64)
    d = Q.shape[1]
    sel = _c(sel, np.int32)
    rows = _c(rows, np.int32)
    n = rows.shape[0]
    O = np.zeros((n, d), dtype=np.float64)
    ds = np.zeros(n, dtype=np.float64)
    lds = np.zeros(n, dtype=np.float64)
    lib().elsaa_oracle_sparse_sets_rows(
        _ptr(Q, _dp), _ptr(K, _dp), _ptr(V, _dp), d, _ptr(sel, _ip),
        sel.shape[1], scale, eps, _ptr(rows, _ip), n, _ptr(O, _dp),
        _ptr(ds, _dp), _ptr(lds, _dp))
    return O, ds, lds


def fuse_rows(O_s, d_s, log_d_s, O_lr, d_lr, lam, g_s, g_lr, eps, mode):
    O_s = _c(O_s, np.float64)
    n, d = O_s.shape
    O = np.zeros((n, d), dtype=np.float64)
    m = np.zeros(n, dtype=np.float64)
    m_log = np.zeros(n, dtype=np.float64)
    args = [_c(a, np.float64) for a in (d_s, log_d_s, O_lr, d_lr, lam, g_s,
                                        g_lr)]
    lib().elsaa_oracle_fuse_rows(n, d, _ptr(O_s, _dp),
                                 *[_ptr(a, _dp) for a in args], eps, mode,
                                 _ptr(O, _dp), _ptr(m, _dp), _ptr(m_log, _dp))
    return O, m, m_log


def dense_rows(Q, K, V, scale, rows=None):
    Q = _c(Q, np.float64)
    K = _c(K, np.float64)
    V = _c(V, np.float64)
    N, d = Q.shape
    if rows is None:
        rows = np.arange(N, dtype=np.int32)
    rows = _c(rows, np.int32)
    O = np.zeros((rows.shape[0], d), dtype=np.float64)
    lds = np.zeros(rows.shape[0], dtype=np.float64)
    lib().elsaa_oracle_dense_rows(_ptr(Q, _dp), _ptr(K, _dp), _ptr(V, _dp),
                                  K.shape[0], d, scale, _ptr(rows, _ip),
                                  rows.shape[0], _ptr(O, _dp), _ptr(lds, _dp))
    return O, lds


# ----------------------------------------------------------- whole operator

def default_params(**kw) -> dict:
    p = dict(block=32, sort_bits=5, gray=1, beta=1.0, eps=1e-6, scale=None,
             lam=1.0, fusion_mode=0)
    p.update(kw)
    return p


def forward_head(q32, k32, v32, w_sort, w_race, p: dict, lam=None,
                 gates=None, rows=None) -> dict:
    """ELSAA for one head (Algorithm 1 steps 4-8 without the projections).

    q32, k32, v32: exact fp32 values [N, d_h]. w_sort [n_s, d_h];
    w_race [L, gamma, d_h]. lam: per-token lambda [N] or None (scalar
    p['lam']). gates: [N, 2] or None (= 1, 1). rows: original query indices
    to evaluate (None = all). Returns fp64 arrays for those rows plus the
    whole-head permutations and keys.
    """
    N, d = q32.shape
    scale = p["scale"] if p.get("scale") else 1.0 / np.sqrt(d)
    # Algorithm sortLSH: hash, sort.
    ws = w_sort if p["sort_bits"] > 0 else np.zeros((0, d), np.float32)
    keys_q, mis_q = sort_keys(q32, ws, p["gray"])
    keys_k, mis_k = sort_keys(k32, ws, p["gray"])
    perm_q = stable_argsort(keys_q)
    perm_k = stable_argsort(keys_k)
    Q = q32.astype(np.float64)
    K = k32.astype(np.float64)
    V = v32.astype(np.float64)
    if rows is None:
        rows = np.arange(N, dtype=np.int32)
    rows = _c(rows, np.int32)
    extra = {}
    if p.get("selector", 0) == 1:
        # top-k selector: block sums, candidate blocks, per-query top-k,
        # then the block step over each query's selected keys
        b = p["block"]
        cand = topk_candidates(block_sums(q32, perm_q, b),
                               block_sums(k32, perm_k, b), p["topk_blocks"])
        sel = topk_select_rows(q32, k32, perm_q, perm_k, b, cand, p["topk"],
                               rows)
        O_s, d_s, log_d_s = sparse_sets_rows(Q, K, V, sel, scale, p["eps"],
                                             rows)
        extra = dict(cand=cand, sel=sel)
    else:
        # Algorithm sortLSH: block attention, un-permuted to the rows.
        O_s, d_s, log_d_s = sortlsh_rows(Q, K, V, perm_q, perm_k, p["block"],
                                         scale, p["eps"], rows,
                                         nb=p.get("neighbors", 0))
    # Algorithm RACE: key-side summaries over all keys, query readout.
    A, Bs = race_summaries(K, V, w_race, p["beta"])
    O_lr, d_lr = race_readout_rows(Q, w_race, p["beta"], p["eps"], A, Bs,
                                   rows)
    # Eq. (5) multiplier and Eq. (6) fusion.
    n = rows.shape[0]
    lam_r = (np.full(n, p["lam"], np.float64) if lam is None
             else _c(lam, np.float64)[rows])
    if gates is None:
        g_s = np.ones(n)
        g_lr = np.ones(n)
    else:
        g = _c(gates, np.float64)
        g_s, g_lr = g[rows, 0], g[rows, 1]
    O, m, m_log = fuse_rows(O_s, d_s, log_d_s, O_lr, d_lr, lam_r, g_s, g_lr,
                            p["eps"], p["fusion_mode"])
    return dict(O=O, O_sparse=O_s, d_sparse=d_s, log_d_sparse=log_d_s,
                O_lr=O_lr, d_lr=d_lr, m=m, m_log=m_log, perm_q=perm_q,
                perm_k=perm_k, keys_q=keys_q, keys_k=keys_k, A=A, B=Bs,
                hash_fp64_mismatch=mis_q + mis_k, rows=rows, **extra)


def params_from_workload(wl, **over) -> dict:
    p = default_params(block=wl.block, sort_bits=wl.sort_bits,
                       gray=wl.gray_order, beta=wl.beta, eps=wl.eps,
                       lam=wl.lam, fusion_mode=wl.fusion_mode)
    p["race_tables"] = wl.race_tables
    p["race_bits"] = wl.race_bits
    p["neighbors"] = getattr(wl, "neighbor_blocks", 0)
    p["causal_chunk"] = getattr(wl, "causal_chunk", 128)
    p["causal_base_len"] = getattr(wl, "causal_base_len", 4096)
    p["selector"] = getattr(wl, "selector", 0)
    p["topk"] = getattr(wl, "topk", 0)
    p["topk_blocks"] = getattr(wl, "topk_blocks", 1)
    p.update(over)
    return p


def forward(inputs: dict, p: dict, lam=None, gates=None, heads=None,
            rows=None, threads: int | None = None) -> dict:
    """ELSAA over [B, H, N, d_h] inputs for the listed (b, h) heads.

    inputs: dict with q, k, v (torch or numpy, any float dtype holding the
    exact input values), w_sort [H, n_s, d_h], w_race [H, L, gamma, d_h].
    heads: list of (b, h) pairs (None = all). rows: query rows per head
    (None = all). Returns {(b, h): forward_head result}.
    """
    q = to_numpy32(inputs["q"])
    k = to_numpy32(inputs["k"])
    v = to_numpy32(inputs["v"])
    w_sort = to_numpy32(inputs["w_sort"])
    w_race = to_numpy32(inputs["w_race"]).astype(np.float64)
    Bn, Hn = q.shape[0], q.shape[1]
    lam_a = None if lam is None else to_numpy32(lam)
    gates_a = None if gates is None else to_numpy32(gates)
    if heads is None:
        heads = [(b, h) for b in range(Bn) for h in range(Hn)]

    def one(bh):
        b, h = bh
        return bh, forward_head(
            q[b, h], k[b, h], v[b, h], w_sort[h], w_race[h], p,
            lam=None if lam_a is None else lam_a[b, h],
            gates=None if gates_a is None else gates_a[b, h], rows=rows)

    threads = threads or min(len(heads), os.cpu_count() or 1)
    if threads <= 1:
        return dict(one(bh) for bh in heads)
    with ThreadPoolExecutor(max_workers=threads) as ex:
        return dict(ex.map(one, heads))
