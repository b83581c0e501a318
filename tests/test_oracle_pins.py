"""Pins for the fp64 oracle: values the paper prints, closed forms, identities,
brute force on tiny inputs and the hardness construction.  CPU only.

Each check is independent of the oracle's own code path (exact rationals,
numpy library routines, the other side of a Lemma 2.1 identity, or a property
of the algorithm), so that a dropped term, a wrong sign or index, or a
transposed operand in the oracle fails at least one of them.
"""
import itertools
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
from tests.conftest import read_golden
from workloads import RowBatch


# ------------------------------------------------------------------ helpers

def single_row_batch(logits, v, k, v_dtype="f32"):
    logits = np.asarray(logits, np.float32).reshape(1, -1)
    v = np.asarray(v, np.float32).reshape(logits.shape[1], -1)
    n, d = v.shape
    k = np.asarray(k, np.int32).reshape(1, -1)
    return RowBatch(rows_per_group=1, d=d, n=np.array([n], np.int32), logits=logits.ravel(),
                    logit_off=np.zeros(1, np.int64), v=v.ravel(), v_off=np.zeros(1, np.int64),
                    v_dtype=v_dtype, k=k, nb=k.shape[1], n_host=np.array([n], np.int32))


def many_rows_batch(L, V, k):
    """L: [rows][n] logits, V: [rows][n][d], k: [rows][nb] or int."""
    L = np.asarray(L, np.float32)
    V = np.asarray(V, np.float32)
    rows, n = L.shape
    d = V.shape[2]
    kk = np.full((rows, 1), k, np.int32) if np.isscalar(k) else np.asarray(k, np.int32)
    return RowBatch(rows_per_group=1, d=d, n=np.full(rows, n, np.int32), logits=L.ravel(),
                    logit_off=np.arange(rows, dtype=np.int64) * n, v=V.ravel(),
                    v_off=np.arange(rows, dtype=np.int64) * n * d, v_dtype="f32", k=kk,
                    nb=kk.shape[1], n_host=np.full(rows, n, np.int32))


def softmax_np(l):
    l = np.asarray(l, np.float64)
    w = np.exp(l - l.max())
    return w / w.sum()


def es_lemma(p, V, members):
    """es(A) by the second form of Lemma 2.1: ||g_A|| / p(A)."""
    mu = p @ V
    A = list(members)
    g = (p[A, None] * (V[A] - mu)).sum(0)
    return float(np.linalg.norm(g) / p[A].sum())


def bits_to_set(words, n):
    return {j for j in range(n) if (int(words[j >> 5]) >> (j & 31)) & 1}


# ------------------------------------------------- values the paper prints

def test_example_2_2_exact_rationals_and_oracle():
    rows, F = read_golden("example_2_2.txt")
    g = {r[0]: r[1:] for r in rows}
    v = [int(x) for x in g["v"]]
    p = [F(x) for x in g["p"]]
    # exact rational recomputation of the printed values (independent of the oracle)
    mu = sum(pi * vi for pi, vi in zip(p, v))

    def es_exact(A):
        pA = sum(p[j] for j in A)
        return abs(sum(p[j] * v[j] for j in A) / pA - mu)

    assert es_exact([int(x) for x in g["topmass_set"]]) == F(g["topmass_gap"][0])
    assert es_exact([int(x) for x in g["best_set"]]) == F(g["ES"][0])
    all_es = {A: es_exact(A) for A in itertools.combinations(range(3), 2)}
    assert min(all_es.values()) == F(g["ES"][0])
    assert F(g["topmass_gap"][0]) / F(g["ES"][0]) == F(g["kappa"][0])

    # oracle on the instance given by masses
    pf = np.array([float(x) for x in p])
    vf = np.array(v, float).reshape(3, 1)
    for A, val in all_es.items():
        mask = np.zeros(3, np.uint8)
        mask[list(A)] = 1
        e = oracle.eval_instance(pf, vf, mask)
        assert e["gap"] == pytest.approx(float(val), rel=1e-14, abs=1e-15)

    # through the logits path: logits = ln p (fp32), the equal masses tie -> lower index
    b = single_row_batch(np.log(pf).astype(np.float32), vf, [2])
    out = oracle.dense_and_topk_gap(b)
    assert bits_to_set(out["kept_bits"][0, 0], 3) == {0, 1}
    assert out["gap"][0, 0] == pytest.approx(0.5, rel=1e-6)
    bs = oracle.best_subset(b)
    assert sorted(bs["best_idx"][0]) == [0, 2]
    assert int(bs["best_rank"][0]) == oracle.colex_rank([0, 2]) == 1
    assert bs["best_gap"][0] == pytest.approx(9 / 22, rel=1e-6)
    assert bs["topk_gap"][0] / bs["best_gap"][0] == pytest.approx(11 / 9, rel=1e-6)
    # the balancing selector reaches ES(2) here with one swap (drop key 1, add key 2)
    sw = oracle.swap_refine(b, E=1)
    assert sw["n_swaps"][0, 0] == 1
    assert (sw["swap_out"][0, 0, 0], sw["swap_in"][0, 0, 0]) == (1, 2)
    assert sw["refined_gap"][0, 0] == pytest.approx(9 / 22, rel=1e-6)


def test_not_submodular_example():
    rows, F = read_golden("not_submodular.txt")
    v = np.array([0.0, 1.0, 2.0, 3.0]).reshape(4, 1)
    p = np.full(4, 0.25)
    for r in rows:
        if r[0] == "mu":
            e = oracle.eval_instance(p, v, np.ones(4, np.uint8))
            assert e["mu"][0] == float(F(r[1]))
            continue
        eq = r.index("=")
        members = [int(x) for x in r[1:eq]]
        val = float(F(r[eq + 1]))
        mask = np.zeros(4, np.uint8)
        mask[members] = 1
        assert oracle.eval_instance(p, v, mask)["gap"] == pytest.approx(val, abs=1e-15)
    # uniform logits pin the tie rule: the top-2 set is {0, 1}
    b = single_row_batch(np.zeros(4, np.float32), v, [2])
    out = oracle.dense_and_topk_gap(b)
    assert bits_to_set(out["kept_bits"][0, 0], 4) == {0, 1}
    assert out["gap"][0, 0] == pytest.approx(1.0, abs=1e-15)  # es({0,1}) = 1


# -------------------------------------------------------------- identities

@pytest.mark.parametrize("seed", range(6))
def test_lemma_identities_and_bound(seed):
    rng = np.random.default_rng(seed)
    n, d = int(rng.integers(3, 40)), int(rng.integers(1, 20))
    logits = (rng.normal(size=n) * rng.uniform(0.2, 4)).astype(np.float32)
    logits[0] += 5
    V = rng.normal(size=(n, d)).astype(np.float32)
    ks = sorted({1, int(rng.integers(1, n)), n - 1 if n > 1 else 1})
    b = single_row_batch(logits, V, ks)
    out = oracle.dense_and_topk_gap(b)
    p = softmax_np(logits)
    Vd = V.astype(np.float64)
    mu = p @ Vd
    np.testing.assert_allclose(out["o"][0], mu, rtol=1e-12, atol=1e-13)
    D = np.max(np.linalg.norm(Vd - mu, axis=1))
    # sum_j p_j (v_j - mu) = 0
    assert np.linalg.norm((p[:, None] * (Vd - mu)).sum(0)) < 1e-12
    order = np.lexsort((np.arange(n), -logits.astype(np.float64)))
    for bi, k in enumerate(ks):
        A = sorted(order[:k].tolist())
        assert bits_to_set(out["kept_bits"][0, bi], n) == set(A)
        gap = out["gap"][0, bi]
        # the three forms of es(A) agree (Lemma 2.1)
        assert out["form1"][0, bi] == pytest.approx(gap, rel=1e-10, abs=1e-13)
        assert out["form2"][0, bi] == pytest.approx(gap, rel=1e-10, abs=1e-13)
        assert es_lemma(p, Vd, A) == pytest.approx(gap, rel=1e-10, abs=1e-13)
        # dropped mass and kept mass
        assert out["dropped"][0, bi] == pytest.approx(1 - p[A].sum(), abs=1e-13)
        assert out["kept_mass"][0, bi] + out["dropped"][0, bi] == pytest.approx(1.0, abs=1e-13)
        assert out["phi"][0, bi] == pytest.approx(gap * out["kept_mass"][0, bi], rel=1e-10, abs=1e-14)
        # es(A*_s) <= 2 D mbar_s
        assert gap <= 2 * D * out["dropped"][0, bi] * (1 + 1e-12) + 1e-15
        # forced-weight output
        np.testing.assert_allclose(out["o_kept"][0, bi], (p[A] @ Vd[A]) / p[A].sum(), rtol=1e-12,
                                   atol=1e-13)


def test_softmax_shift_invariance_and_uniform():
    rng = np.random.default_rng(7)
    n, d = 17, 5
    # logits on a 1/64 grid, so that the shift by 64 is exact in fp32
    l = (np.round(rng.normal(size=n) * 64) / 64).astype(np.float32)
    V = rng.normal(size=(n, d)).astype(np.float32)
    a = oracle.dense_and_topk_gap(single_row_batch(l, V, [4]))
    b = oracle.dense_and_topk_gap(single_row_batch(l + np.float32(64.0), V, [4]))
    assert np.array_equal(l + np.float32(64.0) - np.float32(64.0), l)
    # adding a constant to every logit changes neither p nor anything derived from it
    np.testing.assert_allclose(a["o"], b["o"], rtol=1e-13, atol=1e-15)
    assert a["gap"][0, 0] == pytest.approx(b["gap"][0, 0], rel=1e-12)
    u = oracle.dense_and_topk_gap(single_row_batch(np.zeros(n, np.float32), V, [n]))
    np.testing.assert_allclose(u["o"][0], V.astype(np.float64).mean(0), rtol=1e-13, atol=1e-14)


# ------------------------------------------------------------ special cases

def test_k_equals_n_is_exactly_zero():
    rng = np.random.default_rng(1)
    for n in (1, 2, 5, 33):
        l = rng.normal(size=n).astype(np.float32)
        V = rng.normal(size=(n, 8)).astype(np.float32)
        out = oracle.dense_and_topk_gap(single_row_batch(l, V, [n]))
        assert out["dropped"][0, 0] == 0.0
        np.testing.assert_allclose(out["o_kept"][0, 0], out["o"][0], rtol=1e-14, atol=1e-15)
        assert out["gap"][0, 0] < 1e-14


def test_k_n_minus_1_closed_form():
    # dropping one key j: m_{A^c} = v_j, so es = p_j ||v_j - mu|| / (1 - p_j)  (App. A, remark)
    rng = np.random.default_rng(2)
    for _ in range(5):
        n, d = int(rng.integers(3, 12)), int(rng.integers(1, 9))
        l = (rng.normal(size=n) * 2).astype(np.float32)
        V = rng.normal(size=(n, d)).astype(np.float32)
        p = softmax_np(l)
        Vd = V.astype(np.float64)
        mu = p @ Vd
        closed = p * np.linalg.norm(Vd - mu, axis=1) / (1 - p)
        bs = oracle.best_subset(single_row_batch(l, V, [n - 1]))
        assert bs["best_gap"][0] == pytest.approx(closed.min(), rel=1e-10)
        j = int(np.argmin(closed))
        assert sorted(bs["best_idx"][0]) == [i for i in range(n) if i != j]


def test_k_1_nearest_point():
    rng = np.random.default_rng(3)
    n, d = 10, 4
    l = rng.normal(size=n).astype(np.float32)
    V = rng.normal(size=(n, d)).astype(np.float32)
    p = softmax_np(l)
    mu = p @ V.astype(np.float64)
    dist = np.linalg.norm(V.astype(np.float64) - mu, axis=1)
    bs = oracle.best_subset(single_row_batch(l, V, [1]))
    assert bs["best_gap"][0] == pytest.approx(dist.min(), rel=1e-12)
    assert bs["best_idx"][0][0] == int(np.argmin(dist))


def test_all_values_equal_gap_zero():
    n, d = 9, 6
    rng = np.random.default_rng(4)
    l = rng.normal(size=n).astype(np.float32)
    V = np.tile(rng.normal(size=(1, d)).astype(np.float32), (n, 1))
    out = oracle.dense_and_topk_gap(single_row_batch(l, V, [1, 3, 8]))
    assert np.all(out["gap"] < 1e-14)
    bs = oracle.best_subset(single_row_batch(l, V, [3]))
    assert bs["best_gap"][0] < 1e-14


def test_nonfinite_logit_flags_row():
    l = np.array([0.0, np.inf, 1.0], np.float32)
    V = np.ones((3, 2), np.float32)
    out = oracle.dense_and_topk_gap(single_row_batch(l, V, [1]))
    assert out["status"][0] == 6


# -------------------------------------------------------------- brute force

@pytest.mark.parametrize("seed", range(4))
def test_best_subset_brute_force_small(seed):
    rng = np.random.default_rng(100 + seed)
    rows = 6
    n = int(rng.integers(5, 13))
    d = int(rng.integers(1, 7))
    k = int(rng.integers(1, n + 1))
    L = (rng.normal(size=(rows, n)) * rng.uniform(0.3, 3)).astype(np.float32)
    L[:, 0] += 4
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    bs = oracle.best_subset(many_rows_batch(L, V, k))
    for r in range(rows):
        p = softmax_np(L[r])
        Vd = V[r].astype(np.float64)
        # every mask of size k, scored by the Lemma 2.1 form
        vals = {}
        for mask in range(1 << n):
            if bin(mask).count("1") != k:
                continue
            A = [j for j in range(n) if (mask >> j) & 1]
            vals[tuple(A)] = es_lemma(p, Vd, A)
        best = min(vals.values())
        assert bs["best_gap"][r] == pytest.approx(best, rel=1e-10, abs=1e-14)
        ties = [A for A, e in vals.items() if e <= best * (1 + 1e-12) + 1e-15]
        want = min(ties, key=lambda A: sum(math.comb(c, i + 1) for i, c in enumerate(A)))
        if len(ties) == 1:
            assert tuple(sorted(bs["best_idx"][r])) == want
        others = sorted(vals.values())[1] if len(vals) > 1 else math.inf
        assert bs["second_gap"][r] == pytest.approx(others, rel=1e-10, abs=1e-14)


def test_colex_rank_is_a_bijection_in_colex_order():
    n, k = 9, 4
    combos = list(itertools.combinations(range(n), k))
    colex = sorted(combos, key=lambda c: tuple(reversed(c)))
    assert [oracle.colex_rank(c) for c in colex] == list(range(math.comb(n, k)))


def test_best_le_swap_le_topk_and_random_subsets():
    rng = np.random.default_rng(9)
    rows, n, d, k = 24, 11, 8, 4
    L = (rng.gumbel(size=(rows, n)) * rng.uniform(0.5, 3, size=(rows, 1))).astype(np.float32)
    L[:, 0] += 6
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    b = many_rows_batch(L, V, k)
    bs = oracle.best_subset(b)
    sw = oracle.swap_refine(b, E=n - k)
    rand_med, top_med = [], []
    for r in range(rows):
        p = softmax_np(L[r])
        Vd = V[r].astype(np.float64)
        assert bs["best_gap"][r] <= sw["refined_gap"][r, 0] * (1 + 1e-12)
        assert sw["refined_gap"][r, 0] <= bs["topk_gap"][r] * (1 + 1e-12)
        assert sw["topk_gap"][r, 0] == pytest.approx(bs["topk_gap"][r], rel=1e-12)
        rs = [es_lemma(p, Vd, sorted(rng.choice(n, k, replace=False))) for _ in range(20)]
        assert min(rs) >= bs["best_gap"][r] * (1 - 1e-12)
        rand_med.append(np.median(rs))
        top_med.append(bs["topk_gap"][r])
    # "top-k <= random" holds as a statistic, not per row (Example 2.2 is a counterexample)
    assert np.median(top_med) <= np.median(rand_med)


@pytest.mark.parametrize("seed", range(3))
def test_swap_rule_defining_properties(seed):
    """Every taken swap is the most-decreasing single swap inside the candidate
    set and strictly decreases es; the final set admits no decreasing swap."""
    rng = np.random.default_rng(200 + seed)
    rows, n, d, k, E = 8, 14, 5, 5, 4
    L = (rng.normal(size=(rows, n)) * 1.5).astype(np.float32)
    L[:, 0] += 3
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    sw = oracle.swap_refine(many_rows_batch(L, V, k), E=E)
    for r in range(rows):
        p = softmax_np(L[r])
        Vd = V[r].astype(np.float64)
        mu = p @ Vd
        order = np.lexsort((np.arange(n), -L[r].astype(np.float64)))
        A = set(order[:k].tolist())
        err = p * np.linalg.norm(Vd - mu, axis=1)
        dropped = [j for j in range(n) if j not in A]
        extras = sorted(dropped, key=lambda j: (-err[j], j))[:E]
        pool = A | set(extras)
        cur = es_lemma(p, Vd, sorted(A))
        assert sw["topk_gap"][r, 0] == pytest.approx(cur, rel=1e-12)
        for t in range(int(sw["n_swaps"][r, 0])):
            cand = {(i, j): es_lemma(p, Vd, sorted(A - {i} | {j}))
                    for i in sorted(A) for j in sorted(pool - A)}
            best = min(cand.values())
            i, j = int(sw["swap_out"][r, 0, t]), int(sw["swap_in"][r, 0, t])
            assert cand[(i, j)] == pytest.approx(best, rel=1e-10)
            assert best < cur
            A = A - {i} | {j}
            cur = best
        cand = [es_lemma(p, Vd, sorted(A - {i} | {j})) for i in A for j in pool - A]
        assert not cand or min(cand) >= cur * (1 - 1e-10)
        assert sw["refined_gap"][r, 0] == pytest.approx(cur, rel=1e-10)


# ------------------------------------------------------- hardness construction

def _planted(m, rng, odd=False):
    """App. A.2: d = 1, uniform masses 1/m, integer points, s = m/2."""
    while True:
        w = rng.integers(0, 20, size=m)
        W = int(w.sum())
        if odd:
            if W % 2 == 1:
                return w
            continue
        # plant a balanced split: force sum over the first half = W/2
        half = w[: m // 2].sum()
        rest = w[m // 2:].sum()
        if half == rest:
            perm = rng.permutation(m)
            return w[perm]


@pytest.mark.parametrize("seed", range(3))
def test_hardness_instances(seed):
    rng = np.random.default_rng(300 + seed)
    m = 8
    for odd in (False, True):
        w = _planted(m, rng, odd)
        L = np.zeros((1, m), np.float32)  # uniform masses exactly 1/m
        V = w.astype(np.float32).reshape(1, m, 1)
        bs = oracle.best_subset(many_rows_batch(L, V, m // 2))
        if odd:
            # m^2 g_A is an odd integer's multiple -> ES >= 2/m^2 (Lemma A.5)
            assert bs["best_gap"][0] >= 2.0 / m ** 2 - 1e-12
        else:
            assert bs["best_gap"][0] == 0.0
            A = bs["best_idx"][0]
            assert 2 * int(w[A].sum()) == int(w.sum())


# ---------------------------------------------------------------- ContourKV

def contour_bruteforce(scores, floor, budget, s):
    cells, T = scores.shape
    F = min(floor, T)
    cell_idx, pos_idx = np.meshgrid(np.arange(cells), np.arange(T - F), indexing="ij")
    sc = scores[:, : T - F].astype(np.float64).ravel()
    order = np.lexsort((pos_idx.ravel(), cell_idx.ravel(), -sc))
    K = budget - cells * F
    kept = np.zeros((cells, T), bool)
    kept[:, T - F:] = True
    sel = order[:K]
    kept[cell_idx.ravel()[sel], pos_idx.ravel()[sel]] = True
    tau = sc[order[K - 1]] if K > 0 else math.inf
    counts = kept.sum(1)
    offsets = np.concatenate([[0], np.cumsum(counts)])
    pos = np.concatenate([np.nonzero(kept[h])[0] for h in range(cells)])
    tot = scores.astype(np.float64).sum(1)
    dalloc = np.where(kept, 0, scores).astype(np.float64).sum(1) / tot
    du = []
    for h in range(cells):
        o = np.lexsort((np.arange(T), -scores[h].astype(np.float64)))
        du.append(scores[h][o[s:]].astype(np.float64).sum() / tot[h])
    return counts, offsets, pos, tau, np.array(du), dalloc


@pytest.mark.parametrize("cells,T,floor,frac", [(3, 10, 2, 0.5), (5, 40, 32, 0.9), (4, 64, 8, 0.25),
                                                (2, 7, 32, 1.0)])
def test_contour_alloc_bruteforce(cells, T, floor, frac):
    rng = np.random.default_rng(cells * 100 + T)
    scores = np.exp(rng.normal(size=(cells, T)) * rng.uniform(0.5, 2.5, size=(cells, 1))).astype(np.float32)
    scores[0, :3] = scores[1 % cells, 3]  # ties across cells and positions
    budget = max(cells * min(floor, T), int(frac * cells * T))
    s = budget // cells
    o = oracle.contour_alloc(scores, floor, budget, s)
    assert o["status"] == 0
    c, off, pos, tau, du, da = contour_bruteforce(scores, floor, budget, s)
    np.testing.assert_array_equal(o["counts"], c)
    np.testing.assert_array_equal(o["offsets"], off)
    np.testing.assert_array_equal(o["kept_pos"], pos)
    assert o["offsets"][-1] == budget
    assert np.all(o["counts"] >= min(floor, T))
    assert np.all(np.diff(o["offsets"]) >= 0)
    if math.isfinite(tau):
        assert o["tau"] == np.float32(tau)
    np.testing.assert_allclose(o["dropped_uniform"], du, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(o["dropped_alloc"], da, rtol=1e-12, atol=1e-15)


def test_contour_identical_cells_get_equal_counts():
    rng = np.random.default_rng(5)
    row = np.exp(rng.normal(size=200)).astype(np.float32)
    scores = np.tile(row, (4, 1))
    o = oracle.contour_alloc(scores, 32, 4 * 80, 80)
    # ties break by cell index, so counts differ by at most the tie spill
    assert o["counts"].max() - o["counts"].min() <= 1
    assert oracle.contour_alloc(scores, 32, 4 * 31, 31)["status"] == 1  # below the floors


def test_ragged_compact_bytes():
    rng = np.random.default_rng(6)
    cells, T, d = 3, 20, 8
    K = rng.integers(0, 65535, size=(cells, T, d)).astype(np.uint16)
    V = rng.integers(0, 65535, size=(cells, T, d)).astype(np.uint16)
    scores = rng.random((cells, T)).astype(np.float32)
    o = oracle.contour_alloc(scores, 4, 30, 10)
    Ko, Vo = oracle.ragged_compact(K, V, o["offsets"], o["kept_pos"])
    for h in range(cells):
        a, b = o["offsets"][h], o["offsets"][h + 1]
        np.testing.assert_array_equal(Ko[a:b], K[h, o["kept_pos"][a:b]])
        np.testing.assert_array_equal(Vo[a:b], V[h, o["kept_pos"][a:b]])
