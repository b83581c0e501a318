"""Pins for the decision margins the swap-rule oracle reports, which the GPU
parity tests use to exempt near-ties: the pool-boundary margin of the single-key
errors and the smallest decision margin over the rounds.  A numpy brute force
recomputes both from the definitions (the first round's scores of every
(kept, pool) pair).  CPU only."""
import itertools

import numpy as np
import pytest

import oracle
from tests.test_oracle_pins import many_rows_batch


def first_round(L, V, k, E):
    l = L.astype(np.float32).astype(np.float64)
    p = np.exp(l - l.max())
    p /= p.sum()
    V = V.astype(np.float32).astype(np.float64)
    mu = p @ V
    n = len(p)
    A = list(np.lexsort((np.arange(n), -l))[:k])
    rest = [j for j in range(n) if j not in A]
    err = np.array([p[j] * np.linalg.norm(V[j] - mu) for j in rest])
    order = np.lexsort((np.array(rest), -err))
    pool_x = [rest[t] for t in order[:E]]
    es_sorted = err[order]
    pool_margin = ((es_sorted[E - 1] - es_sorted[E]) / es_sorted[E - 1]) if 0 < E < len(rest) else np.inf

    def es(S):
        S = list(S)
        return np.linalg.norm(p[S] @ V[S] / p[S].sum() - mu)

    cur = es(A)
    scores = sorted(es([a for a in A if a != i] + [j]) for i, j in itertools.product(A, pool_x))
    best = scores[0]
    second = scores[1] if len(scores) > 1 else np.inf
    margin = min((second - best) / cur, abs(cur - best) / cur)
    return pool_margin, margin


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_swap_margins_match_a_brute_force_first_round(seed):
    rng = np.random.default_rng(40 + seed)
    rows, n, d, k, E = 16, 30, 4, 5, 6
    L = rng.normal(size=(rows, n)) * rng.uniform(0.5, 3, size=(rows, 1))
    V = rng.normal(size=(rows, n, d))
    o = oracle.swap_refine(many_rows_batch(L, V, k), E=E, max_swaps=16)
    exact = 0
    for r in range(rows):
        pm, m1 = first_round(L[r], V[r], k, E)
        assert o["pool_margin"][r, 0] == pytest.approx(pm, rel=1e-9, abs=1e-15)
        # the reported margin is the smallest over all rounds: the first round bounds it,
        # and with no swap taken there is only that round
        assert o["margin"][r, 0] <= m1 * (1 + 1e-9) + 1e-15
        if o["n_swaps"][r, 0] == 0:
            assert o["margin"][r, 0] == pytest.approx(m1, rel=1e-9, abs=1e-15)
            exact += 1
    assert o["n_swaps"].max() > 0  # some rows swap, so the bound is exercised too
    assert exact > 0  # and some take none, so the equality is too


def test_every_dropped_key_in_the_pool_has_no_boundary():
    rng = np.random.default_rng(9)
    L = rng.normal(size=(4, 12))
    V = rng.normal(size=(4, 12, 3))
    o = oracle.swap_refine(many_rows_batch(L, V, 4), E=8)
    assert np.all(np.isinf(o["pool_margin"]))


@pytest.mark.parametrize("seed", [0, 1])
def test_swap_scores_match_a_brute_force(seed):
    """orc_swap_scores (every option of one balancing round) against es of
    each swapped set computed from the definition in numpy, on sets that are
    not the top-mass set (so the test does not lean on the selector)."""
    rng = np.random.default_rng(70 + seed)
    rows, n, d = 5, 26, 6
    L = rng.normal(size=(rows, n)) * rng.uniform(0.5, 3, size=(rows, 1))
    V = rng.normal(size=(rows, n, d))
    b = many_rows_batch(L, V, 5)
    for r in range(rows):
        l = L[r].astype(np.float32).astype(np.float64)
        p = np.exp(l - l.max())
        p /= p.sum()
        Vr = V[r].astype(np.float32).astype(np.float64)
        mu = p @ Vr
        A = np.zeros(n, bool)
        A[rng.choice(n, 7, replace=False)] = True
        add = np.flatnonzero(~A)[rng.permutation(n - 7)[:9]]
        got, cur = oracle.swap_scores(b, r, A, add)

        def es(S):
            S = list(S)
            return np.linalg.norm(p[S] @ Vr[S] / p[S].sum() - mu)

        assert cur == pytest.approx(es(np.flatnonzero(A)), rel=1e-12)
        kept = np.flatnonzero(A)
        want = np.array([[es([x for x in kept if x != i] + [j]) for j in add] for i in kept])
        np.testing.assert_allclose(got, want, rtol=1e-11, atol=1e-14)


def test_candidate_set_matches_a_brute_force():
    """orc_candidate_set: the top-mass set plus the E dropped keys of largest
    p_j ||v_j - mu|| (Definition 2.2), ties to the lower index; boundary margin."""
    rng = np.random.default_rng(81)
    rows, n, d, k = 6, 30, 5, 6
    L = rng.normal(size=(rows, n)) * rng.uniform(0.5, 3, size=(rows, 1))
    L[0, 3:9] = L[0, 3]  # a tie in the logits at the budget boundary
    V = rng.normal(size=(rows, n, d))
    b = many_rows_batch(L, V, k)
    for r in range(rows):
        for E in (0, 1, 5, n - k, n):
            l = L[r].astype(np.float32).astype(np.float64)
            p = np.exp(l - l.max())
            p /= p.sum()
            Vr = V[r].astype(np.float32).astype(np.float64)
            mu = p @ Vr
            A = list(np.lexsort((np.arange(n), -l))[:k])
            rest = [j for j in range(n) if j not in A]
            err = np.array([p[j] * np.linalg.norm(Vr[j] - mu) for j in rest])
            order = np.lexsort((np.array(rest), -err))
            want = sorted(A + [rest[t] for t in order[:E]])
            pool, pm = oracle.candidate_set(b, r, k, E)
            np.testing.assert_array_equal(pool, want)
            if 0 < E < len(rest):
                es_sorted = err[order]
                assert pm == pytest.approx((es_sorted[E - 1] - es_sorted[E]) / es_sorted[E - 1], rel=1e-9, abs=1e-15)
            else:
                assert np.isinf(pm)
