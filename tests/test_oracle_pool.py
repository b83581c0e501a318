"""Pins for the oracle's candidate-set search ES_pool (Definition 2.2: the exact
best size-s subset of the top-mass set plus the E dropped keys of largest
single-key error).  CPU only.

Each check stands outside the function under test: Example 2.2's printed
values, the plain exhaustive search (a different oracle function) when the
pool is every key, a brute force that builds the pool and scores subsets by
the second form of Lemma 2.1 in numpy, the order ES <= ES_pool <= es(balancing)
<= es(top-mass) that Definition 2.2 and the balancing selector imply, and exact
ties that only the tie rule decides.
"""
import itertools

import numpy as np
import pytest

import oracle
from tests.conftest import read_golden
from tests.test_oracle_pins import many_rows_batch, single_row_batch


def test_example_2_2_pool_is_every_key():
    # s = 2 with one extra: the candidate set is all three keys, so ES_pool(2)
    # = ES(2) = 9/22 at {1, 3} (0-based {0, 2}) and kappa-hat = 11/9
    rows, F = read_golden("example_2_2.txt")
    g = {r[0]: r[1:] for r in rows}
    p = np.array([float(F(x)) for x in g["p"]])
    v = np.array([int(x) for x in g["v"]], float).reshape(3, 1)
    b = single_row_batch(np.log(p).astype(np.float32), v, [2])
    o = oracle.pool_best_subset(b, E=[1])
    assert o["call_status"] == 0 and o["n_subsets"][0, 0] == 3
    assert sorted(o["best_idx"][0, 0]) == [int(x) for x in g["best_set"]]
    assert o["best_gap"][0, 0] == pytest.approx(float(F(g["ES"][0])), rel=1e-6)
    assert o["topk_gap"][0, 0] / o["best_gap"][0, 0] == pytest.approx(float(F(g["kappa"][0])), rel=1e-6)
    # with no extras the pool is the top-mass set itself
    o0 = oracle.pool_best_subset(b, E=[0])
    assert o0["n_subsets"][0, 0] == 1 and sorted(o0["best_idx"][0, 0]) == [0, 1]
    assert o0["best_gap"][0, 0] == pytest.approx(0.5, rel=1e-6)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_full_pool_equals_exhaustive_search(seed):
    # E >= n - s puts every key in the pool: ES_pool = ES of the plain search
    rng = np.random.default_rng(seed)
    rows, n, d = 12, 13, 5
    L = rng.normal(size=(rows, n)) * rng.uniform(0.5, 3, size=(rows, 1))
    V = rng.normal(size=(rows, n, d))
    k = rng.integers(1, n, size=(rows, 1))
    b = many_rows_batch(L, V, k)
    o = oracle.pool_best_subset(b, E=[n])
    assert np.all(np.isinf(o["pool_margin"]))  # every dropped key joins: no pool boundary
    es = oracle.best_subset(b)
    np.testing.assert_allclose(o["best_gap"][:, 0], es["best_gap"], rtol=1e-12, atol=1e-15)
    for r in range(rows):
        if es["second_gap"][r] - es["best_gap"][r] > 1e-9 * es["best_gap"][r]:
            assert sorted(o["best_idx"][r, 0][:k[r, 0]]) == sorted(es["best_idx"][r][:k[r, 0]])


def _brute_pool(L, V, s, E):
    """Build the candidate set in numpy and score every size-s subset of it by
    es = ||g_A|| / p(A) (Lemma 2.1).  Returns (best es, best set, es(top-mass),
    relative margin between the E-th and (E+1)-th single-key errors)."""
    l = L.astype(np.float32).astype(np.float64)
    p = np.exp(l - l.max())
    p /= p.sum()
    V = V.astype(np.float32).astype(np.float64)
    mu = p @ V
    n = len(p)
    top = sorted(np.lexsort((np.arange(n), -l))[:s])
    rest = [j for j in range(n) if j not in top]
    err = np.array([p[j] * np.linalg.norm(V[j] - mu) for j in rest])
    extras = [rest[t] for t in np.lexsort((np.array(rest), -err))[:E]]
    pool = sorted(top + extras)

    def es(A):
        A = list(A)
        g = (p[A, None] * (V[A] - mu)).sum(0)
        return np.linalg.norm(g) / p[A].sum()

    best = min((es(A), A) for A in itertools.combinations(pool, s))
    e_sorted = np.sort(err)[::-1]
    margin = (e_sorted[E - 1] - e_sorted[E]) / e_sorted[E - 1] if 0 < E < len(rest) else np.inf
    return best[0], list(best[1]), es(top), margin


@pytest.mark.parametrize("s,E", [(3, 4), (5, 6), (2, 9)])
def test_brute_force_over_the_pool(s, E):
    rng = np.random.default_rng(100 + s)
    rows, n, d = 6, 40, 4
    L = rng.normal(size=(rows, n)) * 2.0
    V = rng.normal(size=(rows, n, d))
    b = many_rows_batch(L, V, s)
    o = oracle.pool_best_subset(b, E=[E])
    for r in range(rows):
        best, A, top, margin = _brute_pool(L[r], V[r], s, E)
        assert o["best_gap"][r, 0] == pytest.approx(best, rel=1e-10, abs=1e-14)
        assert o["pool_margin"][r, 0] == pytest.approx(margin, rel=1e-9, abs=1e-15)
        assert o["topk_gap"][r, 0] == pytest.approx(top, rel=1e-10, abs=1e-14)
        if o["second_gap"][r, 0] - best > 1e-9 * best:
            assert list(o["best_idx"][r, 0]) == A


@pytest.mark.parametrize("seed", [0, 1])
def test_order_es_le_pool_le_balancing_le_top_mass(seed):
    # a larger set of subsets can only lower the minimum; the balancing selector
    # moves inside the same candidate set and starts from the top-mass set
    rng = np.random.default_rng(7 + seed)
    rows, n, d = 10, 14, 3
    L = rng.normal(size=(rows, n)) * 1.5
    V = rng.normal(size=(rows, n, d))
    s, E = 4, 3
    b = many_rows_batch(L, V, s)
    o = oracle.pool_best_subset(b, E=[E])
    es = oracle.best_subset(b)
    sw = oracle.swap_refine(b, E=E)
    tol = 1e-12
    assert np.all(es["best_gap"] <= o["best_gap"][:, 0] * (1 + tol) + 1e-15)
    assert np.all(o["best_gap"][:, 0] <= sw["refined_gap"][:, 0] * (1 + tol) + 1e-15)
    assert np.all(sw["refined_gap"][:, 0] <= o["topk_gap"][:, 0] * (1 + tol) + 1e-15)
    np.testing.assert_allclose(o["n_subsets"][:, 0], 35)  # C(4 + 3, 4)


def test_exact_ties_take_the_smallest_colex_rank():
    # uniform masses, v = (-3, -1, 1, 3): mu = 0 and {0, 3}, {1, 2} both give
    # es = 0 exactly.  Lexicographic order meets {0, 3} first; colex rank
    # prefers {1, 2} (C(1,1) + C(2,2) = 2 < C(0,1) + C(3,2) = 3)
    b = single_row_batch(np.zeros(4, np.float32), np.array([[-3.0], [-1.0], [1.0], [3.0]]), [2])
    o = oracle.pool_best_subset(b, E=[2])
    assert o["n_subsets"][0, 0] == 6
    assert list(o["best_idx"][0, 0]) == [1, 2]
    assert o["best_gap"][0, 0] == 0.0 and o["second_gap"][0, 0] == 0.0
    assert list(oracle.best_subset(b)["best_idx"][0]) == [1, 2]  # the same rule as the plain search


def test_paper_schedule_subset_counts_and_arguments():
    # 24 / 12 / 6 / 4 extras at s = 4 / 8 / 16 / 32 give C(28,4), C(20,8),
    # C(22,16) and C(36,32) subsets per instance
    rng = np.random.default_rng(3)
    n, d = 200, 2
    L = rng.normal(size=(1, n)).astype(np.float32)
    V = rng.normal(size=(1, n, d))
    b = many_rows_batch(L, V, np.array([[4, 8, 16, 32]]))
    o = oracle.pool_best_subset(b, E=[24, 12, 6, 4], max_subsets=1)
    assert list(o["n_subsets"][0]) == [20475, 125970, 74613, 58905]
    assert o["call_status"] != 0  # over the subset cap: refused
    b2 = many_rows_batch(L, V, np.array([[4, 8]]))
    o2 = oracle.pool_best_subset(b2, E=[24, 12])
    assert o2["call_status"] == 0
    assert np.all(o2["best_gap"][0] <= o2["topk_gap"][0])
