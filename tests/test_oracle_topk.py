"""Pins of the top-k selector in the oracle (oracle/elsaa_oracle.c, steps 1-4
of the selector reading; Section 3 names per-query top-k selection as a
future selector and defines none). CPU only.

* a hand-worked case (tests/golden/topk_n8.txt): block sums, candidate
  blocks and selected key sets, ties included;
* integer-valued inputs, where every fp32 chain is exact: candidates and
  key sets equal a brute-force numpy ranking (np.lexsort on the exact
  integer scores, lower index first among ties), many ties included;
* c = 1, k = b: each query keeps its whole sorted block, so the branch equals
  the sorted-block branch (Algorithm sortLSH);
* c = N / b, k = N: every key is kept, so with eps = 0 the branch is dense
  softmax attention (Eq. (1)-(2));
* invariants: k distinct keys per query, all from the query's candidate
  blocks.
"""
import os

import numpy as np
import pytest

from oracle import oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def read_golden():
    vals = {}
    with open(os.path.join(GOLDEN, "topk_n8.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                key, val = line.split(":")
                vals[key] = np.array([int(x) for x in val.split()])
    return vals


def test_hand_worked_example():
    g = read_golden()
    q = g["q"].reshape(8, 2).astype(np.float32)
    k = g["k"].reshape(8, 2).astype(np.float32)
    ident = np.arange(8, dtype=np.int32)
    qs = orc.block_sums(q, ident, 2)
    ks = orc.block_sums(k, ident, 2)
    np.testing.assert_array_equal(qs, [[2, 1], [-1, 1], [1, -2], [2, 0]])
    np.testing.assert_array_equal(ks, [[1, 1], [-1, -1], [0, 0], [2, 2]])
    cand = orc.topk_candidates(qs, ks, 2)
    np.testing.assert_array_equal(cand, g["cand"].reshape(4, 2))
    sel = orc.topk_select_rows(q, k, ident, ident, 2, cand, 2, ident)
    np.testing.assert_array_equal(sel, g["sel"].reshape(8, 2))


def brute_force(q, k, perm_q, perm_k, b, c, topk):
    """Exact integer ranking with numpy (inputs are small integers, so the
    oracle's fp32 chains are exact and must agree)."""
    N = q.shape[0]
    T = N // b
    qi = q.astype(np.int64)
    ki = k.astype(np.int64)
    qsum = np.stack([qi[perm_q[t * b:(t + 1) * b]].sum(0) for t in range(T)])
    ksum = np.stack([ki[perm_k[u * b:(u + 1) * b]].sum(0) for u in range(T)])
    s = qsum @ ksum.T
    cand = np.zeros((T, c), np.int64)
    for t in range(T):
        others = np.array([u for u in range(T) if u != t])
        order = others[np.lexsort((others, -s[t, others]))]
        cand[t] = [t] + list(order[:c - 1])
    sel = np.zeros((N, topk), np.int64)
    pos = np.argsort(perm_q)
    for i in range(N):
        t = pos[i] // b
        keys = np.concatenate([perm_k[u * b:(u + 1) * b] for u in cand[t]])
        sc = ki[keys] @ qi[i]
        keep = keys[np.lexsort((keys, -sc))[:topk]]
        sel[i] = np.sort(keep)
    return cand, sel


@pytest.mark.parametrize("N,d,b,c,topk,lim,seed", [
    (64, 4, 8, 2, 8, 2, 0), (64, 4, 8, 3, 5, 1, 1), (96, 6, 16, 2, 20, 2, 2),
    (128, 8, 32, 4, 32, 3, 3), (48, 3, 8, 6, 48, 1, 4), (64, 4, 16, 1, 7, 2, 5),
])
def test_integer_inputs_match_brute_force(N, d, b, c, topk, lim, seed):
    rng = np.random.default_rng(seed)
    q = rng.integers(-lim, lim + 1, (N, d)).astype(np.float32)
    k = rng.integers(-lim, lim + 1, (N, d)).astype(np.float32)
    perm_q = rng.permutation(N).astype(np.int32)
    perm_k = rng.permutation(N).astype(np.int32)
    want_cand, want_sel = brute_force(q, k, perm_q, perm_k, b, c, topk)
    cand = orc.topk_candidates(orc.block_sums(q, perm_q, b),
                               orc.block_sums(k, perm_k, b), c)
    np.testing.assert_array_equal(cand, want_cand)
    sel = orc.topk_select_rows(q, k, perm_q, perm_k, b, cand, topk,
                               np.arange(N, dtype=np.int32))
    np.testing.assert_array_equal(sel, want_sel)


def _head(N, d, seed):
    rng = np.random.default_rng(seed)
    q = (2 * rng.standard_normal((N, d))).astype(np.float32)
    k = rng.standard_normal((N, d)).astype(np.float32)
    v = rng.standard_normal((N, d)).astype(np.float32)
    w_sort = rng.standard_normal((5, d)).astype(np.float32)
    w_race = rng.standard_normal((4, 4, d))
    return q, k, v, w_sort, w_race


@pytest.mark.parametrize("N,d,b", [(256, 16, 32), (192, 8, 64)])
def test_one_block_whole_budget_is_the_sorted_block_branch(N, d, b):
    q, k, v, w_sort, w_race = _head(N, d, 7)
    base = orc.default_params(block=b)
    ref = orc.forward_head(q, k, v, w_sort, w_race, base)
    got = orc.forward_head(q, k, v, w_sort, w_race,
                           dict(base, selector=1, topk=b, topk_blocks=1))
    pos = np.argsort(ref["perm_q"])
    for i in range(N):
        t = pos[i] // b
        want = np.sort(ref["perm_k"][t * b:(t + 1) * b])
        np.testing.assert_array_equal(got["sel"][i], want)
    for name in ("O_sparse", "log_d_sparse", "O"):
        np.testing.assert_allclose(got[name], ref[name], rtol=0, atol=1e-12)


def test_every_block_whole_sequence_is_dense_attention():
    N, d, b = 96, 8, 16
    q, k, v, w_sort, w_race = _head(N, d, 8)
    p = orc.default_params(block=b, eps=0.0, selector=1, topk=N,
                           topk_blocks=N // b)
    got = orc.forward_head(q, k, v, w_sort, w_race, p)
    O, logd = orc.dense_rows(q.astype(np.float64), k.astype(np.float64),
                             v.astype(np.float64), 1.0 / np.sqrt(d))
    np.testing.assert_allclose(got["O_sparse"], O, rtol=0, atol=1e-12)
    np.testing.assert_allclose(got["log_d_sparse"], logd, rtol=0, atol=1e-12)


def test_selected_sets_are_valid():
    N, d, b, c, topk = 256, 16, 32, 3, 40
    q, k, v, w_sort, w_race = _head(N, d, 9)
    p = orc.default_params(block=b, selector=1, topk=topk, topk_blocks=c)
    r = orc.forward_head(q, k, v, w_sort, w_race, p)
    pos = np.argsort(r["perm_q"])
    assert (r["cand"][:, 0] == np.arange(N // b)).all()
    for t in range(N // b):
        assert len(set(r["cand"][t].tolist())) == c
    for i in range(N):
        s = r["sel"][i]
        assert len(set(s.tolist())) == topk and (np.diff(s) > 0).all()
        allowed = np.concatenate([r["perm_k"][u * b:(u + 1) * b]
                                  for u in r["cand"][pos[i] // b]])
        assert set(s.tolist()) <= set(allowed.tolist())
    assert np.isfinite(r["O"]).all()
