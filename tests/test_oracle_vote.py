"""Pins for the oracle's group vote (f1: one kept set per KV head, the s keys of
largest mass summed over the head's query rows, Sec. 2.1).  CPU only.

Each check stands outside the oracle's own code path: a worked example in
exact rationals, exact ties that only the tie rule decides, the paper's
statement that a group of one row reproduces the row's own top-mass set (a
different ranking -- by logit -- in a different oracle function), identical
rows, and the per-row optimum ES(s) found by brute force as a lower bound.
"""
import itertools
from fractions import Fraction

import numpy as np
import pytest

import oracle
from workloads import RowBatch


def group_batch(L, V, s):
    """L: [groups][rows_per_group][n] logits, V: [groups][n][d] values shared
    by the group's rows, s: [groups][nb] budgets (also used as the rows' k)."""
    L = np.asarray(L, np.float32)
    V = np.asarray(V, np.float32)
    G, R, n = L.shape
    d = V.shape[2]
    s = np.asarray(s, np.int32).reshape(G, -1)
    k = np.repeat(s, R, axis=0)
    return RowBatch(rows_per_group=R, d=d, n=np.full(G, n, np.int32), logits=L.ravel(),
                    logit_off=np.arange(G, dtype=np.int64) * R * n, v=V.ravel(),
                    v_off=np.arange(G, dtype=np.int64) * n * d, v_dtype="f32", k=k, nb=k.shape[1],
                    n_host=np.full(G, n, np.int32))


def members(words, n):
    return [j for j in range(n) if (int(words[j >> 5]) >> (j & 31)) & 1]


def test_worked_example_exact_rationals():
    # Two rows share v = (-1, 1, 5) (d = 1): p1 = (1/2, 3/10, 1/5),
    # p2 = (1/10, 1/5, 7/10).  Summed mass G = (3/5, 1/2, 9/10), so the vote
    # keeps {2} at s = 1 and {0, 2} at s = 2.
    P = [[Fraction(1, 2), Fraction(3, 10), Fraction(1, 5)], [Fraction(1, 10), Fraction(1, 5), Fraction(7, 10)]]
    v = [Fraction(-1), Fraction(1), Fraction(5)]

    def es(p, A):
        mu = sum(pj * vj for pj, vj in zip(p, v))
        pa = sum(p[j] for j in A)
        return abs(sum(p[j] * v[j] for j in A) / pa - mu), 1 - pa

    # the numbers worked by hand: row 1 keeps {0, 2}: m_A = 5/7, mu = 4/5,
    # es = 3/35; row 2: m_A = 17/4, mu = 18/5, es = 13/20.
    assert es(P[0], [0, 2]) == (Fraction(3, 35), Fraction(3, 10))
    assert es(P[1], [0, 2]) == (Fraction(13, 20), Fraction(1, 5))
    assert es(P[0], [2]) == (Fraction(21, 5), Fraction(4, 5))
    assert es(P[1], [2]) == (Fraction(7, 5), Fraction(3, 10))
    L = np.log(np.array([[float(x) for x in row] for row in P]))[None]
    b = group_batch(L, np.array([[[-1.0], [1.0], [5.0]]]), [[1, 2, 3]])
    o = oracle.group_vote(b, b.k[:1])
    assert members(o["bits"][0, 0], 3) == [2]
    assert members(o["bits"][0, 1], 3) == [0, 2]
    assert members(o["bits"][0, 2], 3) == [0, 1, 2]
    want_gap = [[21 / 5, 3 / 35, 0.0], [7 / 5, 13 / 20, 0.0]]
    want_drop = [[4 / 5, 3 / 10, 0.0], [3 / 10, 1 / 5, 0.0]]
    np.testing.assert_allclose(o["gap"], want_gap, rtol=1e-6, atol=1e-7)
    np.testing.assert_allclose(o["dropped"], want_drop, rtol=1e-6, atol=1e-7)
    # s = n: the complement is empty, so the dropped mass is exactly 0 (es is 0
    # up to the rounding of m_A = N_A / p(A))
    assert (o["dropped"][:, 2] == 0.0).all() and (o["gap"][:, 2] < 1e-14).all()
    np.testing.assert_allclose(o["mass"][0], [0.6, 0.5, 0.9], rtol=1e-6)
    # margins: (9/10 - 3/5) / (9/10) at s = 1, (3/5 - 1/2) / (3/5) at s = 2, 1 at s = n
    np.testing.assert_allclose(o["margin"][0], [1 / 3, 1 / 6, 1.0], rtol=1e-6)
    assert (o["status"] == 0).all()
    # against their own top-mass sets the vote helps row 1 ({0, 1}: es 21/20)
    # and costs row 2 ({1, 2}: es 23/45)
    own = oracle.dense_and_topk_gap(b)
    np.testing.assert_allclose(own["gap"][:, 1], [21 / 20, 23 / 45], rtol=1e-6)


def test_exact_ties_keep_lower_indices():
    # uniform logits: every p_j is the same double, so G ties exactly at every
    # key and only the tie rule decides the set
    n, R = 7, 3
    L = np.zeros((2, R, n))
    V = np.random.default_rng(0).normal(size=(2, n, 4))
    o = oracle.group_vote(group_batch(L, V, [[1, 3, 7], [2, 5, 6]]), [[1, 3, 7], [2, 5, 6]])
    for g, ss in enumerate([[1, 3, 7], [2, 5, 6]]):
        for b, s in enumerate(ss):
            assert members(o["bits"][g, b], n) == list(range(s))
            assert o["margin"][g, b] == (1.0 if s == n else 0.0)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_group_of_one_is_the_rows_own_top_mass_set(seed):
    # with one row per group the summed mass is the row's own p, so the vote
    # is the row's own top-mass set (Sec. 2.1); the oracle ranks that one by
    # logit in a separate function
    rng = np.random.default_rng(seed)
    rows, n, d = 40, 50, 8
    L = rng.normal(size=(rows, 1, n)) * rng.uniform(0.5, 3.0, size=(rows, 1, 1))
    V = rng.normal(size=(rows, n, d))
    s = rng.integers(1, n + 1, size=(rows, 3))
    b = group_batch(L, V, s)
    o = oracle.group_vote(b, s)
    own = oracle.dense_and_topk_gap(b)
    np.testing.assert_array_equal(o["bits"], own["kept_bits"])
    np.testing.assert_allclose(o["gap"], own["gap"], rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(o["dropped"], own["dropped"], rtol=1e-12, atol=1e-15)


def test_identical_rows_vote_like_one_row():
    # R copies of one row: G = R p keeps the order of p, so every row keeps its
    # own top-mass set
    rng = np.random.default_rng(4)
    G, R, n, d = 6, 5, 33, 16
    L = np.repeat(rng.normal(size=(G, 1, n)) * 2, R, axis=1)
    V = rng.normal(size=(G, n, d))
    s = rng.integers(1, n + 1, size=(G, 2))
    b = group_batch(L, V, s)
    o = oracle.group_vote(b, s)
    own = oracle.dense_and_topk_gap(b)
    for g in range(G):
        for i in range(R):
            np.testing.assert_array_equal(o["bits"][g], own["kept_bits"][g * R + i])
    np.testing.assert_allclose(o["gap"], own["gap"], rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("seed", [0, 1])
def test_per_row_optimum_lower_bounds_the_vote(seed):
    # every row could have kept the shared set itself, so ES(s) of each row
    # (brute force over all size-s subsets) is at most the vote's es
    rng = np.random.default_rng(10 + seed)
    G, R, n, d, s = 4, 4, 10, 3, 4
    L = rng.normal(size=(G, R, n)) * 1.5
    V = rng.normal(size=(G, n, d))
    b = group_batch(L, V, np.full((G, 1), s))
    o = oracle.group_vote(b, np.full((G, 1), s))
    for g in range(G):
        for i in range(R):
            lw = L[g, i].astype(np.float32).astype(np.float64)
            p = np.exp(lw - lw.max())
            p /= p.sum()
            mu = p @ V[g].astype(np.float32)
            best = min(np.linalg.norm(p[list(A)] @ V[g].astype(np.float32)[list(A)] / p[list(A)].sum() - mu)
                       for A in itertools.combinations(range(n), s))
            assert best <= o["gap"][g * R + i, 0] * (1 + 1e-12) + 1e-15


def test_out_of_range_budget_and_nonfinite_flag_the_group():
    rng = np.random.default_rng(3)
    L = rng.normal(size=(3, 2, 6))
    L[2, 1, 4] = np.inf
    V = rng.normal(size=(3, 6, 2))
    s = np.array([[2], [7], [3]])
    o = oracle.group_vote(group_batch(L, V, np.minimum(s, 6)), s)
    assert list(o["status"]) == [0, 0, 1, 1, 6, 6]


def test_eval_mask_skips_rows_but_not_the_vote():
    rng = np.random.default_rng(8)
    L = rng.normal(size=(2, 3, 20)) * 2
    V = rng.normal(size=(2, 20, 4))
    s = np.array([[5], [9]])
    b = group_batch(L, V, s)
    full = oracle.group_vote(b, s)
    part = oracle.group_vote(b, s, eval_rows=np.array([1, 0, 1, 0, 0, 1], bool))
    np.testing.assert_array_equal(full["bits"], part["bits"])
    np.testing.assert_array_equal(full["gap"][[0, 2, 5]], part["gap"][[0, 2, 5]])
    assert (part["gap"][[1, 3, 4]] == 0).all()
