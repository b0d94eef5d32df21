"""Pins of the CPU oracle against facts the paper and the mathematics fix.

Every check here computes its expectation by an independent route (a
textbook routine in numpy/scipy, a closed form, a brute-force N x N matrix, a
hand-worked value), never by re-typing the oracle's own loop. Runs on CPU.
"""
import json
import os

import numpy as np
import pytest
from scipy.special import logsumexp, softmax, expit

from oracle import oracle as orc
from paper_2607_20214_gb300 import perfmodel

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rand_head(N, d, seed, temp=1.0, dtype=np.float32):
    rng = np.random.default_rng(seed)
    q = (rng.standard_normal((N, d)) * temp).astype(dtype)
    k = rng.standard_normal((N, d)).astype(dtype)
    v = rng.standard_normal((N, d)).astype(dtype)
    return q, k, v


def planes(d, n_s, L, gamma, seed):
    rng = np.random.default_rng(seed + 100)
    w_sort = rng.standard_normal((n_s, d)).astype(np.float32)
    w_race = rng.standard_normal((L, gamma, d))
    return w_sort, w_race


def np_phi(x, w_race, beta):
    """RACE features by the product identity (independent of the oracle's
    literal softmax): phi_r = prod_b sigmoid(2 beta u_b v_rb)."""
    L, gamma, _ = w_race.shape
    R = 1 << gamma
    u = np.tanh(np.einsum("lgd,nd->nlg", w_race, x))  # [n, L, gamma]
    s = expit(2.0 * beta * u)
    corners = np.array([[1.0 if (r >> b) & 1 else -1.0 for b in range(gamma)]
                        for r in range(R)])  # [R, gamma]
    pos = corners > 0
    fac = np.where(pos[None, None], s[:, :, None, :], 1.0 - s[:, :, None, :])
    return fac.prod(axis=-1)  # [n, L, R]


# ------------------------------------------------------------- the hash

def test_sort_keys_hand_built_2d():
    # d = 2, planes = unit axes, so bit 0 = [x > 0], bit 1 = [y > 0].
    w = np.array([[1, 0], [0, 1]], np.float32)
    x = np.array([[1, 1], [-1, 1], [-1, -1], [1, -1], [0, 1], [0, 0]],
                 np.float32)
    # codes: 3, 2, 0, 1, 2 (zero projection is not > 0), 0
    keys_bin, _ = orc.sort_keys(x, w, gray=0)
    assert keys_bin.tolist() == [3, 2, 0, 1, 2, 0]
    # Gray rank of codes 0,1,2,3 in the sequence 0,1,3,2 is 0,1,3,2.
    keys_gray, _ = orc.sort_keys(x, w, gray=1)
    assert keys_gray.tolist() == [2, 3, 0, 1, 3, 0]


def test_gray_rank_matches_reflected_gray_sequence():
    n_s = 5
    d = n_s
    w = np.eye(n_s, dtype=np.float32)
    codes = np.arange(1 << n_s)
    x = np.array([[1.0 if (c >> p) & 1 else -1.0 for p in range(n_s)]
                  for c in codes], np.float32)
    keys, _ = orc.sort_keys(x, w, gray=1)
    seq = [k ^ (k >> 1) for k in range(1 << n_s)]  # reflected Gray sequence
    expect = [seq.index(c) for c in codes]
    assert keys.tolist() == expect
    # neighbours in sort order differ in exactly one hash bit
    order = np.argsort(keys)
    for a, b in zip(codes[order][:-1], codes[order][1:]):
        assert bin(int(a) ^ int(b)).count("1") == 1


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_sort_keys_match_fp64_signs(seed):
    q, _, _ = rand_head(512, 64, seed, temp=2.0)
    w, _ = planes(64, 5, 1, 1, seed)
    keys, mism = orc.sort_keys(q, w, gray=0)
    proj = q.astype(np.float64) @ w.astype(np.float64).T
    ok = np.abs(proj).min(axis=1) > 1e-3  # away from the sign boundary
    codes = ((proj > 0) * (1 << np.arange(5))).sum(axis=1)
    assert np.array_equal(keys[ok], codes[ok])
    assert mism == 0


def test_zero_sort_bits_gives_identity_order():
    q, _, _ = rand_head(100, 8, 3)
    keys, _ = orc.sort_keys(q, np.zeros((0, 8), np.float32), gray=1)
    assert not keys.any()
    assert np.array_equal(orc.stable_argsort(keys), np.arange(100))


# ------------------------------------------------------------- the sort

@pytest.mark.parametrize("N,nbins", [(1, 4), (7, 2), (1000, 32), (4099, 3)])
def test_stable_argsort_matches_numpy_stable(N, nbins):
    rng = np.random.default_rng(N)
    keys = rng.integers(0, nbins, N).astype(np.uint16)
    perm = orc.stable_argsort(keys)
    assert np.array_equal(perm, np.argsort(keys, kind="stable"))
    # validity: bijection, keys non-decreasing, ties by increasing index
    assert np.array_equal(np.sort(perm), np.arange(N))
    ks = keys[perm]
    assert np.all(np.diff(ks.astype(int)) >= 0)
    tie = np.diff(ks.astype(int)) == 0
    assert np.all(np.diff(perm)[tie] > 0)


def test_duplicate_keys_share_codes_and_keep_index_order():
    q, k, _ = rand_head(256, 32, 9)
    k[128:192] = k[0:64]
    w, _ = planes(32, 5, 1, 1, 9)
    keys, _ = orc.sort_keys(k, w, gray=1)
    assert np.array_equal(keys[128:192], keys[0:64])
    perm = orc.stable_argsort(keys)
    pos = np.empty_like(perm)
    pos[perm] = np.arange(256)
    assert np.all(pos[0:64] < pos[128:192])


# ---------------------------------------------------- the sparse branch

@pytest.mark.parametrize("N,d,seed", [(64, 16, 0), (128, 32, 1), (96, 8, 2)])
def test_single_block_is_dense_softmax_attention(N, d, seed):
    """b = N: one block holds every key, so the branch is Eq. (2) exactly."""
    q, k, v = rand_head(N, d, seed, temp=2.0)
    w_sort, w_race = planes(d, 5, 2, 3, seed)
    p = orc.default_params(block=N, eps=0.0)
    res = orc.forward_head(q, k, v, w_sort, w_race, p)
    z = (q.astype(np.float64) @ k.astype(np.float64).T) / np.sqrt(d)
    o_ref = softmax(z, axis=1) @ v.astype(np.float64)
    np.testing.assert_allclose(res["O_sparse"], o_ref, rtol=1e-12,
                               atol=1e-12)
    np.testing.assert_allclose(res["log_d_sparse"], logsumexp(z, axis=1),
                               rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("b", [8, 16, 32])
def test_zero_sort_bits_is_block_diagonal_local_attention(b):
    """n_s = 0: identity order, so query i attends to keys of block i // b."""
    N, d = 96, 16
    q, k, v = rand_head(N, d, b, temp=1.5)
    _, w_race = planes(d, 0, 2, 2, b)
    p = orc.default_params(block=b, sort_bits=0, eps=1e-6)
    res = orc.forward_head(q, k, v, np.zeros((0, d), np.float32), w_race, p)
    z = (q.astype(np.float64) @ k.astype(np.float64).T) / np.sqrt(d)
    blk = np.arange(N) // b
    z_masked = np.where(blk[:, None] == blk[None, :], z, -np.inf)
    e = np.exp(z_masked)
    den = e.sum(axis=1)
    o_ref = (e @ v.astype(np.float64)) / (den + 1e-6)[:, None]
    np.testing.assert_allclose(res["O_sparse"], o_ref, rtol=1e-11,
                               atol=1e-12)
    np.testing.assert_allclose(res["d_sparse"], den, rtol=1e-12)


@pytest.mark.parametrize("b,nb", [(16, 1), (8, 2), (32, 1)])
def test_neighbour_blocks_with_zero_sort_bits_are_banded(b, nb):
    """n_s = 0 and nb neighbouring blocks: query i attends to the keys of
    blocks i // b - nb .. i // b + nb (clipped at the ends), brute force."""
    N, d = 96, 16
    q, k, v = rand_head(N, d, b + nb, temp=1.5)
    _, w_race = planes(d, 0, 2, 2, b)
    p = orc.default_params(block=b, sort_bits=0, eps=1e-6, neighbors=nb)
    res = orc.forward_head(q, k, v, np.zeros((0, d), np.float32), w_race, p)
    z = (q.astype(np.float64) @ k.astype(np.float64).T) / np.sqrt(d)
    blk = np.arange(N) // b
    band = np.abs(blk[:, None] - blk[None, :]) <= nb
    e = np.exp(np.where(band, z, -np.inf))
    den = e.sum(axis=1)
    o_ref = (e @ v.astype(np.float64)) / (den + 1e-6)[:, None]
    np.testing.assert_allclose(res["O_sparse"], o_ref, rtol=1e-11,
                               atol=1e-12)
    np.testing.assert_allclose(res["d_sparse"], den, rtol=1e-12)
    # the first and last blocks see nb fewer blocks than the middle ones
    assert band[0].sum() == (nb + 1) * b
    assert band[N // 2].sum() == min(N, (2 * nb + 1) * b)


def test_neighbour_blocks_covering_all_blocks_give_dense_attention():
    """nb >= N / b - 1: every query attends to all N keys, whatever the
    hash and the sort (dense softmax attention, scipy)."""
    N, d, b = 64, 16, 16
    q, k, v = rand_head(N, d, 9, temp=2.0)
    w_sort, w_race = planes(d, 5, 2, 2, 9)
    p = orc.default_params(block=b, sort_bits=5, eps=0.0,
                           neighbors=N // b - 1)
    res = orc.forward_head(q, k, v, w_sort, w_race, p)
    z = (q.astype(np.float64) @ k.astype(np.float64).T) / np.sqrt(d)
    np.testing.assert_allclose(res["O_sparse"],
                               softmax(z, axis=1) @ v.astype(np.float64),
                               rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(np.log(res["d_sparse"]),
                               logsumexp(z, axis=1), rtol=1e-12)


def test_query_block_t_attends_exactly_key_block_t():
    """V = identity: sparse weights of query i are nonzero exactly on the
    keys of its block (query block t <-> key block t of the sorted orders)."""
    N = d = 32
    b = 8
    q, k, _ = rand_head(N, d, 5, temp=1.0)
    v = np.eye(N, dtype=np.float32)
    w_sort, w_race = planes(d, 3, 1, 2, 5)
    p = orc.default_params(block=b, sort_bits=3, eps=1e-6)
    res = orc.forward_head(q, k, v, w_sort, w_race, p)
    perm_q = np.argsort(res["keys_q"], kind="stable")
    perm_k = np.argsort(res["keys_k"], kind="stable")
    pos_q = np.empty(N, int)
    pos_q[perm_q] = np.arange(N)
    for i in range(N):
        t = pos_q[i] // b
        support = set(perm_k[t * b:(t + 1) * b].tolist())
        nz = set(np.nonzero(res["O_sparse"][i] > 0)[0].tolist())
        assert nz == support
        # row weights of the sparse branch sum to d_s / (d_s + eps)
        ds = res["d_sparse"][i]
        assert res["O_sparse"][i].sum() == pytest.approx(ds / (ds + 1e-6),
                                                         rel=1e-12)


# ------------------------------------------------------- the RACE branch

def test_race_feature_softmax_equals_product_identity():
    rng = np.random.default_rng(4)
    w = rng.standard_normal((3, 4, 16))
    for beta in (0.3, 1.0, 5.0):
        for _ in range(5):
            x = rng.standard_normal(16)
            phi = orc.race_features(x, w, beta)
            np.testing.assert_allclose(phi, np_phi(x[None], w, beta)[0],
                                       rtol=1e-12, atol=1e-15)
            np.testing.assert_allclose(phi.sum(axis=1), 1.0, rtol=1e-13)


def test_race_beta_zero_closed_form():
    """beta = 0: phi = 1/R, A_r = N/R, Den = N/R,
    O_lr = (N/R)/(N/R + eps) * mean_j V_j."""
    N, d, L, gamma, eps = 200, 12, 3, 3, 1e-6
    q, k, v = rand_head(N, d, 11)
    _, w_race = planes(d, 0, L, gamma, 11)
    R = 1 << gamma
    A, Bs = orc.race_summaries(k, v, w_race, 0.0)
    np.testing.assert_allclose(A, N / R, rtol=1e-13)
    rows = np.arange(N, dtype=np.int32)
    O, dlr = orc.race_readout_rows(q, w_race, 0.0, eps, A, Bs, rows)
    np.testing.assert_allclose(dlr, N / R, rtol=1e-13)
    expect = (N / R) / (N / R + eps) * v.astype(np.float64).mean(axis=0)
    np.testing.assert_allclose(O, np.broadcast_to(expect, O.shape),
                               rtol=1e-11, atol=1e-14)


@pytest.mark.parametrize("beta", [0.5, 1.0, 3.0])
def test_race_matches_brute_force_kernel_matrix(beta):
    """O_lr,i = sum_j kappa_ij V_j / (sum_j kappa_ij + eps) with the explicit
    N x N kernel kappa_ij = (1/L) sum_l phi^l(Q_i) . phi^l(K_j)."""
    N, d, L, gamma, eps = 150, 10, 4, 3, 1e-6
    q, k, v = rand_head(N, d, 21, temp=0.5)
    _, w_race = planes(d, 0, L, gamma, 21)
    w_race = w_race * 0.3
    A, Bs = orc.race_summaries(k, v, w_race, beta)
    O, dlr = orc.race_readout_rows(q, w_race, beta, eps, A, Bs,
                                   np.arange(N, dtype=np.int32))
    pq = np_phi(q.astype(np.float64), w_race, beta)
    pk = np_phi(k.astype(np.float64), w_race, beta)
    kappa = np.einsum("ilr,jlr->ij", pq, pk) / L
    den = kappa.sum(axis=1)
    o_ref = kappa @ v.astype(np.float64) / (den + eps)[:, None]
    np.testing.assert_allclose(dlr, den, rtol=1e-12)
    np.testing.assert_allclose(O, o_ref, rtol=1e-10, atol=1e-13)
    # invariants: sum_r A^l_r = N, 0 < d_lr <= N
    np.testing.assert_allclose(A.sum(axis=1), N, rtol=1e-13)
    assert np.all(dlr > 0) and np.all(dlr <= N * (1 + 1e-12))


def test_race_large_beta_counts_bucket_collisions():
    """beta -> infinity: one-hot buckets, Den_i = mean over tables of the
    number of keys that share query i's hypercube corner."""
    N, d, L, gamma = 120, 6, 3, 2
    q, k, v = rand_head(N, d, 31)
    _, w_race = planes(d, 0, L, gamma, 31)
    A, Bs = orc.race_summaries(k, v, w_race, 1e4)
    _, dlr = orc.race_readout_rows(q, w_race, 1e4, 1e-6, A, Bs,
                                   np.arange(N, dtype=np.int32))
    pw = 1 << np.arange(gamma)
    bq = ((np.einsum("lgd,nd->nlg", w_race, q.astype(np.float64)) > 0)
          * pw).sum(-1)
    bk = ((np.einsum("lgd,nd->nlg", w_race, k.astype(np.float64)) > 0)
          * pw).sum(-1)
    counts = (bq[:, None, :] == bk[None, :, :]).sum(axis=1).mean(axis=1)
    np.testing.assert_allclose(dlr, counts, rtol=1e-5, atol=1e-5)


def test_race_hand_worked_one_dim():
    """d_h = 1, gamma = 1, L = 1, w = 1, beta = 1.
    phi(x) = (1 - s, s) with s = sigmoid(2 tanh x). Keys 0 and big x:
    phi(0) = (1/2, 1/2); phi(x -> inf) -> (1 - sigmoid(2), sigmoid(2))."""
    w = np.ones((1, 1, 1))
    K = np.array([[0.0], [50.0]])
    V = np.array([[2.0], [-1.0]])
    A, Bs = orc.race_summaries(K, V, w, 1.0)
    s2 = 1.0 / (1.0 + np.exp(-2.0))
    np.testing.assert_allclose(A[0], [0.5 + (1 - s2), 0.5 + s2], rtol=1e-13)
    np.testing.assert_allclose(Bs[0, :, 0], [1.0 - (1 - s2), 1.0 - s2],
                               rtol=1e-13)
    O, dlr = orc.race_readout_rows(np.array([[0.0]]), w, 1.0, 0.0, A, Bs,
                                   np.array([0], np.int32))
    # query at 0 reads the bucket average: Den = (A0 + A1)/2 = 1
    np.testing.assert_allclose(dlr, [1.0], rtol=1e-13)
    np.testing.assert_allclose(O[0, 0], (Bs[0, 0, 0] + Bs[0, 1, 0]) / 2,
                               rtol=1e-13)


# --------------------------------------------------------------- fusion

def _full(N=64, d=16, b=16, seed=0, **kw):
    q, k, v = rand_head(N, d, seed, temp=2.0)
    w_sort, w_race = planes(d, 4, 2, 3, seed)
    p = orc.default_params(block=b, sort_bits=4, **kw)
    return q, k, v, w_sort, w_race, p


def test_multiplier_direct_equals_log_domain_and_in_unit_interval():
    q, k, v, ws, wr, p = _full()
    rng = np.random.default_rng(0)
    lam = rng.uniform(0.3, 1.8, 64)
    res = orc.forward_head(q, k, v, ws, wr, p, lam=lam)
    np.testing.assert_allclose(res["m"], res["m_log"], rtol=1e-12)
    assert np.all(res["m"] > 0) and np.all(res["m"] < 1)
    expect = res["d_sparse"] / (res["d_sparse"] + lam * res["d_lr"] + 1e-6)
    np.testing.assert_allclose(res["m"], expect, rtol=1e-13)


def test_gates_select_branches_and_ablation_sets_m_to_one():
    q, k, v, ws, wr, p = _full(seed=3)
    N = q.shape[0]
    only_lr = np.tile([0.0, 1.0], (N, 1))
    res = orc.forward_head(q, k, v, ws, wr, p, gates=only_lr)
    np.testing.assert_allclose(res["O"], res["O_lr"], rtol=0, atol=0)
    gates = np.random.default_rng(1).uniform(0.05, 0.95, (N, 2))
    p1 = dict(p, fusion_mode=1)
    res1 = orc.forward_head(q, k, v, ws, wr, p1, gates=gates)
    assert np.all(res1["m"] == 1.0)
    np.testing.assert_allclose(
        res1["O"], gates[:, :1] * res1["O_sparse"] + gates[:, 1:] *
        res1["O_lr"], rtol=1e-14, atol=1e-15)


def test_lambda_zero_single_block_gives_dense_attention():
    N, d = 48, 8
    q, k, v = rand_head(N, d, 2, temp=2.0)
    ws, wr = planes(d, 4, 2, 2, 2)
    p = orc.default_params(block=N, sort_bits=4, eps=1e-300)
    gates = np.tile([1.0, 0.0], (N, 1))
    res = orc.forward_head(q, k, v, ws, wr, p, lam=np.zeros(N), gates=gates)
    z = (q.astype(np.float64) @ k.astype(np.float64).T) / np.sqrt(d)
    np.testing.assert_allclose(res["O"], softmax(z, axis=1) @ v, rtol=1e-12,
                               atol=1e-13)


def test_convex_value_weights():
    """V = identity exposes the weights of O_i = sum_j w_ij V_j: w >= 0 and
    sum_j w_ij = g_s m d_s/(d_s+eps) + g_lr Den/(Den+eps)."""
    N = d = 48
    q, k, _ = rand_head(N, d, 8, temp=2.0)
    v = np.eye(N, dtype=np.float32)
    ws, wr = planes(d, 3, 2, 3, 8)
    gates = np.random.default_rng(2).uniform(0.05, 0.95, (N, 2))
    p = orc.default_params(block=12, sort_bits=3)
    res = orc.forward_head(q, k, v, ws, wr, p, gates=gates)
    W = res["O"]
    assert np.all(W >= 0)
    eps = 1e-6
    ds, dl = res["d_sparse"], res["d_lr"]
    expect = gates[:, 0] * res["m"] * ds / (ds + eps) + gates[:, 1] * dl / (
        dl + eps)
    np.testing.assert_allclose(W.sum(axis=1), expect, rtol=1e-12)


# -------------------------------------------------------- paper numbers

def test_interaction_counts_match_appendix_f():
    g = json.load(open(os.path.join(GOLDEN, "complexity_example.json")))
    c = perfmodel.interaction_counts(**{"N": g["inputs"]["N"],
                                        "s": g["inputs"]["s"],
                                        "L_s": g["inputs"]["L_s"],
                                        "gamma": g["inputs"]["gamma"]})
    for key in ("full", "sparse", "race", "elsaa"):
        assert c[key] == g[key]
    assert round(100 * c["sparse"] / c["full"], 1) == \
        g["sparse_percent_of_full"]
    assert round(100 * c["race"] / c["full"], 1) == g["race_percent_of_full"]
    assert round(100 * c["elsaa"] / c["full"], 1) == \
        g["elsaa_percent_of_full"]
