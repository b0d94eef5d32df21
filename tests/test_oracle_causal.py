"""Pins of the causal oracle (oracle/causal.py). CPU only.

Causal sparse branch (Algorithm "Causal sortLSH", CausalSparse / SortLSH /
MergeLSE):
* n <= N0: exact causal attention = dense softmax over each row's prefix
  (the C oracle's dense rows on K[:i+1]), eps = 0;
* one block covering every half (b >= N) and eps = 0: the recursion merges
  disjoint key sets exactly, so CausalSparse is exact causal attention for
  every N0 < N, odd lengths (padding) included;
* the attended key set of every row equals the set worked out by hand
  for N = 8 (tests/golden/causal_sets_*.txt: one code for all rows, distinct
  codes, tied codes), and for larger cases with one code the set built from
  the split rule; with eps = 0 the output is softmax attention over that
  set;
* MergeLSE of two disjoint pieces = attention over their union (eps = 0);
* keys and values after row i never reach row i.
Causal RACE (Algorithm "Causal RACE"):
* the chunked algorithm equals the kernel form
  O_i = sum_{j<=i} k_ij V_j / (sum_{j<=i} k_ij + eps),
  k_ij = (1/L) sum_l phi_l(Q_i) . phi_l(K_j), for chunk sizes that do and do
  not divide N;
* beta = 0: phi = 1/R, d_lr,i = (i + 1)/R, O_lr,i = prefix mean scaled;
* the last row sees every key: equals the non-causal RACE readout.
Planted mistakes in a copy of causal.py each fail one of these pins.
"""
import importlib.util
import os

import numpy as np
import pytest

from oracle import causal as oc
from oracle import oracle as orc

_GD = os.path.join(os.path.dirname(__file__), "golden")
# (file, N0, b): hand-derived key sets, optionally with the rows' codes
GOLDEN_SETS = [("causal_sets_n8.txt", 2, 2),
               ("causal_sets_codes_n8.txt", 4, 2),
               ("causal_sets_ties_n8.txt", 4, 2)]


def read_golden_sets(name):
    codes = {}
    sets = {}
    with open(os.path.join(_GD, name)) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if not line:
                continue
            key, val = line.split(":")
            if key.startswith("codes_"):
                codes[key[6:]] = np.array([int(x) for x in val.split()],
                                          np.uint16)
            else:
                sets[int(key)] = set(int(x) for x in val.split())
    return codes, sets


def _qkv(n, d=8, seed=0, temp=1.0):
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((n, d)) * temp, rng.standard_normal((n, d)),
            rng.standard_normal((n, d)))


def _dense_prefix(Q, K, V, scale):
    """Row i: softmax attention over keys 0..i (C oracle's dense rows)."""
    n, d = Q.shape
    O = np.zeros((n, d))
    ld = np.zeros(n)
    for i in range(n):
        o, l = orc.dense_rows(Q[i:i + 1], K[:i + 1], V[:i + 1], scale)
        O[i], ld[i] = o[0], l[0]
    return O, ld


def _attend_sets(mod, n, hq, hk, pad_code, b, N0):
    """Recover each row's key set by running CausalSparse on one-hot values
    with equal scores (Q = 0): O_i is uniform over the attended keys."""
    V = np.eye(n)
    O, _ = mod.causal_sparse(np.zeros((n, n)), np.zeros((n, n)), V, hq, hk,
                             pad_code, b, N0, 1.0, 0.0)
    return [set(np.nonzero(O[i] > 1e-12)[0].tolist()) for i in range(n)]


def _split_rule_sets(n, b, N0):
    """Key sets of the recursion with one code for every row (the stable
    sort keeps list order), built from the split rule on lists of row
    indices (-1 = padding row): a row attends its base segment's prefix
    and, at every node where it lies in the future half, the past-half
    block with its block index."""
    sets = [set() for _ in range(n)]

    def rec(rows):
        if len(rows) <= N0:
            for a, i in enumerate(rows):
                if i >= 0:
                    sets[i] |= {j for j in rows[:a + 1] if j >= 0}
            return
        if len(rows) % 2:
            rows = rows + [-1]
        m = len(rows) // 2
        past, fut = rows[:m], rows[m:]
        rec(past)
        rec(fut)
        for t, i in enumerate(fut):
            if i >= 0:
                blk = past[(t // b) * b:(t // b + 1) * b]
                sets[i] |= {j for j in blk if j >= 0}

    rec(list(range(n)))
    return sets


def _trace_sets(mod, n, hq, hk, b, N0):
    """Each row's key set rebuilt from the SortLSH orders the recursion
    records (its trace) alone: the row's base-segment prefix, plus at every
    recorded call the past-half keys of the block holding the row's sorted
    position. Needs n = n_leaf 2^k (no padding)."""
    trace = []
    Q = np.zeros((n, 2))
    mod.causal_sparse(Q, Q, Q, hq, hk, 0, b, N0, 1.0, 0.0, trace)
    leaf = n
    while leaf > N0:
        leaf //= 2
    sets = [set(range(i - i % leaf, i + 1)) for i in range(n)]
    for _, _, qrows, krows in trace:
        for p, i in enumerate(qrows):
            t = p // b
            sets[int(i)] |= set(int(j) for j in krows[t * b:(t + 1) * b])
    return sets


def check_sparse_pins(mod):
    scale = 0.7
    # (1) n <= N0: exact causal attention
    Q, K, V = _qkv(37, seed=1, temp=2.0)
    h = np.zeros(37, np.uint16)
    O, ld = mod.causal_sparse(Q, K, V, h, h, 0, 4, 64, scale, 0.0)
    Od, ldd = _dense_prefix(Q, K, V, scale)
    np.testing.assert_allclose(O, Od, rtol=0, atol=1e-12)
    np.testing.assert_allclose(ld, ldd, rtol=0, atol=1e-12)
    # (2) one block everywhere: exact causal attention through the recursion
    for n, N0 in [(40, 8), (37, 5), (33, 1), (64, 16)]:
        Q, K, V = _qkv(n, seed=n, temp=1.5)
        rng = np.random.default_rng(n)
        hq = rng.integers(0, 32, n).astype(np.uint16)
        hk = rng.integers(0, 32, n).astype(np.uint16)
        O, ld = mod.causal_sparse(Q, K, V, hq, hk, 0, 4 * n, N0, scale, 0.0)
        Od, ldd = _dense_prefix(Q, K, V, scale)
        np.testing.assert_allclose(O, Od, rtol=0, atol=1e-11)
        np.testing.assert_allclose(ld, ldd, rtol=0, atol=1e-11)
    # (3) the hand-written sets (tests/golden/causal_sets_*.txt)
    for name, N0, b in GOLDEN_SETS:
        codes, want = read_golden_sets(name)
        z8 = np.zeros(8, np.uint16)
        got = _attend_sets(mod, 8, codes.get("q", z8), codes.get("k", z8), 0,
                           b, N0)
        for i, ks in want.items():
            assert got[i] == ks, (name, i, got[i], ks)
        # the recorded sorted orders give the same sets
        got = _trace_sets(mod, 8, codes.get("q", z8), codes.get("k", z8), b,
                          N0)
        for i, ks in want.items():
            assert got[i] == ks, (name, "trace", i, got[i], ks)
    for n, b, N0 in [(64, 8, 8), (50, 4, 6), (41, 8, 5), (96, 16, 12)]:
        zn = np.zeros(n, np.uint16)
        assert _attend_sets(mod, n, zn, zn, 0, b, N0) == \
            _split_rule_sets(n, b, N0), (n, b, N0)
    for n, b, N0 in [(64, 8, 8), (96, 16, 12)]:
        zn = np.zeros(n, np.uint16)
        assert _trace_sets(mod, n, zn, zn, b, N0) == \
            _split_rule_sets(n, b, N0), (n, b, N0)
    # with random codes: the trace's orders are stable argsorts of each
    # half's codes, and rebuild the sets the one-hot run shows
    rng = np.random.default_rng(17)
    n, b, N0 = 64, 4, 8
    hq = rng.integers(0, 4, n).astype(np.uint16)
    hk = rng.integers(0, 4, n).astype(np.uint16)
    trace = []
    Q = np.zeros((n, 2))
    mod.causal_sparse(Q, Q, Q, hq, hk, 0, b, N0, 1.0, 0.0, trace)
    assert sorted((t[0], t[1]) for t in trace) == [
        (1, 0), (2, 0), (2, 32), (3, 0), (3, 16), (3, 32), (3, 48)]
    for level, start, qrows, krows in trace:
        m = n >> level
        fut = np.arange(start + m, start + 2 * m)
        past = np.arange(start, start + m)
        np.testing.assert_array_equal(
            qrows, fut[np.argsort(hq[fut], kind="stable")])
        np.testing.assert_array_equal(
            krows, past[np.argsort(hk[past], kind="stable")])
    assert _trace_sets(mod, n, hq, hk, b, N0) == \
        _attend_sets(mod, n, hq, hk, 0, b, N0)
    # ... and with real scores, softmax over exactly those sets
    n, b, N0 = 50, 4, 6
    Q, K, V = _qkv(n, seed=5, temp=2.0)
    zn = np.zeros(n, np.uint16)
    O, ld = mod.causal_sparse(Q, K, V, zn, zn, 0, b, N0, scale, 0.0)
    for i, ks in enumerate(_split_rule_sets(n, b, N0)):
        ks = sorted(ks)
        o, l = orc.dense_rows(Q[i:i + 1], K[ks], V[ks], scale)
        np.testing.assert_allclose(O[i], o[0], rtol=0, atol=1e-12)
        assert abs(ld[i] - l[0]) < 1e-12
    # (4) MergeLSE of disjoint pieces = attention over the union
    Q, K, V = _qkv(6, seed=9)
    o1, l1 = orc.dense_rows(Q, K[:3], V[:3], scale)
    o2, l2 = orc.dense_rows(Q, K[3:], V[3:], scale)
    o, l = mod.merge_lse(o1, l1, o2, l2, 0.0)
    ou, lu = orc.dense_rows(Q, K, V, scale)
    np.testing.assert_allclose(o, ou, rtol=0, atol=1e-13)
    np.testing.assert_allclose(l, lu, rtol=0, atol=1e-13)
    # epsilon enters as written: O = (w1 O1 + w2 O2) / (s + eps)
    o, l = mod.merge_lse(np.ones((1, 2)), np.zeros(1), np.ones((1, 2)),
                         np.zeros(1), 0.5)
    np.testing.assert_allclose(o, [[2 / 2.5, 2 / 2.5]], atol=1e-15)
    assert abs(l[0] - np.log(2.5)) < 1e-15
    # (5) later keys and values never reach earlier rows
    n, b, N0 = 48, 4, 6
    Q, K, V = _qkv(n, seed=11)
    rng = np.random.default_rng(3)
    hq = rng.integers(0, 8, n).astype(np.uint16)
    hk = rng.integers(0, 8, n).astype(np.uint16)
    O, _ = mod.causal_sparse(Q, K, V, hq, hk, 0, b, N0, scale, 1e-6)
    K2, V2 = K.copy(), V.copy()
    K2[30:] += 5.0
    V2[30:] -= 3.0
    O2, _ = mod.causal_sparse(Q, K2, V2, hq, hk, 0, b, N0, scale, 1e-6)
    np.testing.assert_array_equal(O[:30], O2[:30])
    assert np.abs(O[30:] - O2[30:]).max() > 1e-3


def _kernel_form(Q, K, V, w_race, beta, eps):
    pQ = oc.race_features_rows(Q, w_race, beta)
    pK = oc.race_features_rows(K, w_race, beta)
    L = pQ.shape[1]
    kap = np.einsum("ilr,jlr->ij", pQ, pK) / L
    kap = np.tril(kap)
    den = kap.sum(axis=1)
    return (kap @ V) / (den + eps)[:, None], den


def check_race_pins(mod):
    rng = np.random.default_rng(2)
    N, d, L, g = 45, 6, 3, 3
    Q = rng.standard_normal((N, d))
    K = rng.standard_normal((N, d))
    V = rng.standard_normal((N, d))
    w = rng.standard_normal((L, g, d))
    Ok, dk = _kernel_form(Q, K, V, w, 1.3, 1e-6)
    for C in (1, 4, 7, 16, 45, 64):
        O, dl = mod.causal_race(Q, K, V, w, 1.3, C, 1e-6)
        np.testing.assert_allclose(O, Ok, rtol=0, atol=1e-12)
        np.testing.assert_allclose(dl, dk, rtol=1e-12, atol=0)
    # beta = 0: phi = 1/R
    R = 1 << g
    O, dl = mod.causal_race(Q, K, V, w, 0.0, 8, 1e-6)
    i = np.arange(N)
    np.testing.assert_allclose(dl, (i + 1) / R, rtol=1e-13)
    want = (np.cumsum(V, axis=0) / R) / ((i + 1) / R + 1e-6)[:, None]
    np.testing.assert_allclose(O, want, rtol=0, atol=1e-12)
    # the last row sees every key: the non-causal RACE readout
    A, Bs = orc.race_summaries(K, V, w, 1.3)
    On, dn = orc.race_readout_rows(Q, w, 1.3, 1e-6, A, Bs,
                                   np.array([N - 1], np.int32))
    O, dl = mod.causal_race(Q, K, V, w, 1.3, 16, 1e-6)
    np.testing.assert_allclose(O[-1], On[0], rtol=0, atol=1e-12)
    assert abs(dl[-1] - dn[0]) < 1e-12 * dn[0]


def test_causal_sparse_pins():
    check_sparse_pins(oc)


def test_causal_race_pins():
    check_race_pins(oc)


def test_golden_sets_match_split_rule():
    """The hand-written N = 8 sets agree with the split-rule construction
    (two independent statements of the same recursion)."""
    _, want = read_golden_sets("causal_sets_n8.txt")
    rule = _split_rule_sets(8, 2, 2)
    for i, ks in want.items():
        assert rule[i] == ks


def test_forward_head_fusion():
    """The whole causal operator: the fusion of the two causal branches
    with the log-domain multiplier; the first row sees only itself."""
    rng = np.random.default_rng(4)
    N, d = 40, 8
    q = rng.standard_normal((N, d)).astype(np.float32)
    k = rng.standard_normal((N, d)).astype(np.float32)
    v = rng.standard_normal((N, d)).astype(np.float32)
    ws = rng.standard_normal((3, d)).astype(np.float32)
    wr = rng.standard_normal((2, 3, d))
    p = orc.default_params(block=4, sort_bits=3, causal_chunk=8,
                           causal_base_len=6)
    r = oc.forward_head(q, k, v, ws, wr, p)
    assert np.isfinite(r["O"]).all()
    m = r["m_log"]
    assert np.all((m > 0) & (m < 1))
    want = m[:, None] * r["O_sparse"] + r["O_lr"]
    np.testing.assert_allclose(r["O"], want, rtol=0, atol=1e-12)
    # row 0 attends only key 0 in both branches
    np.testing.assert_allclose(r["O_sparse"][0],
                               v[0] * np.exp(r["log_d_sparse"][0]) /
                               (np.exp(r["log_d_sparse"][0]) + 1e-6),
                               rtol=1e-12)
    np.testing.assert_allclose(r["O_lr"][0],
                               v[0] * r["d_lr"][0] / (r["d_lr"][0] + 1e-6),
                               rtol=1e-12)


MUTATIONS = [
    ("inclusive_prefix", "sA[1:] = np.cumsum(A, axis=0)[:-1]",
     "sA[:] = np.cumsum(A, axis=0)"),
    ("prefix_B_not_shifted", "sB[1:] = np.cumsum(B, axis=0)[:-1]",
     "sB[:] = np.cumsum(B, axis=0)"),
    ("upper_triangle", "tril = np.tril(np.ones((C, C)))",
     "tril = np.triu(np.ones((C, C)))"),
    ("strict_lower_triangle", "tril = np.tril(np.ones((C, C)))",
     "tril = np.tril(np.ones((C, C)), -1)"),
    ("table_average_dropped",
     "Mn = sum(pQ[sl, l] @ pK[sl, l].T for l in range(L)) / L * tril",
     "Mn = sum(pQ[sl, l] @ pK[sl, l].T for l in range(L)) * tril"),
    ("merge_weights_swapped",
     "O = (w1[:, None] * O1 + w2[:, None] * O2) / (s + eps)[:, None]",
     "O = (w2[:, None] * O1 + w1[:, None] * O2) / (s + eps)[:, None]"),
    ("merge_log_drops_max", "return O, mu + np.log(s + eps)",
     "return O, np.log(s + eps)"),
    ("off_block_reads_future_keys",
     "O_off, ld_off = sortlsh_pair(Q[m:], K[:m], V[:m], hq[m:], hk[:m], b,",
     "O_off, ld_off = sortlsh_pair(Q[m:], K[m:], V[m:], hq[m:], hk[m:], b,"),
    ("base_case_not_causal", "z[np.triu_indices(n, 1)] = -np.inf",
     "pass"),
    ("key_order_unsorted", "pk = orc.stable_argsort(hk)",
     "pk = np.arange(m)"),
    ("split_uneven", "m = n // 2", "m = n // 2 + 1"),
]


@pytest.mark.parametrize("name,old,new", MUTATIONS,
                         ids=[m[0] for m in MUTATIONS])
def test_planted_causal_mistake_is_caught(tmp_path, name, old, new):
    src = open(oc.__file__).read()
    assert src.count(old) == 1, name
    path = tmp_path / "mutant_causal.py"
    path.write_text(src.replace(old, new).replace(
        "from . import oracle as orc", "from oracle import oracle as orc"))
    spec = importlib.util.spec_from_file_location("mutant_causal", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    # a mutant fails a pin (an assertion) or cannot run at all (a split
    # that never shrinks recurses without end)
    with pytest.raises((AssertionError, RecursionError)):
        check_sparse_pins(mod)
        check_race_pins(mod)
