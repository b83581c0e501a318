"""Pins for the enforced-budget ContourKV oracle (Sec. 4: enforcement caps
every head at a uniform method's per-head count): a numpy brute force of the
allocation followed by the per-cell truncation, the cap that truncates
nothing, and the cap equal to the floor.  CPU only."""
import math

import numpy as np
import pytest

import oracle
from tests.test_oracle_pins import contour_bruteforce


def capped_bruteforce(scores, floor, budget, s, cap):
    cells, T = scores.shape
    F = min(floor, T)
    c, off, pos, tau, du, _ = contour_bruteforce(scores, floor, budget, s)
    kept = np.zeros((cells, T), bool)
    for h in range(cells):
        mine = pos[off[h]:off[h + 1]]
        nf = mine[mine < T - F]
        order = np.lexsort((nf, -scores[h, nf].astype(np.float64)))
        kept[h, nf[order[: cap - F]]] = True
        kept[h, T - F:] = True
    counts = kept.sum(1)
    offsets = np.concatenate([[0], np.cumsum(counts)])
    kpos = np.concatenate([np.nonzero(kept[h])[0] for h in range(cells)])
    tot = scores.astype(np.float64).sum(1)
    da = np.where(kept, 0, scores).astype(np.float64).sum(1) / tot
    return counts, offsets, kpos, tau, du, da, c


@pytest.mark.parametrize("cells,T,floor,frac,cap", [(3, 10, 2, 0.5, 4), (5, 40, 32, 0.9, 35), (4, 64, 8, 0.25, 12),
                                                    (6, 50, 4, 0.6, 30), (2, 7, 32, 1.0, 7)])
def test_capped_matches_a_brute_force(cells, T, floor, frac, cap):
    rng = np.random.default_rng(cells * 10 + T + cap)
    scores = np.exp(rng.normal(size=(cells, T)) * rng.uniform(0.5, 2.5, size=(cells, 1))).astype(np.float32)
    scores[0, :3] = scores[1 % cells, 3]  # ties across cells and positions
    budget = max(cells * min(floor, T), int(frac * cells * T))
    s = budget // cells
    o = oracle.contour_alloc_capped(scores, floor, budget, s, cap)
    assert o["status"] == 0
    counts, offsets, kpos, tau, du, da, c0 = capped_bruteforce(scores, floor, budget, s, cap)
    np.testing.assert_array_equal(o["counts"], counts)
    np.testing.assert_array_equal(o["counts"], np.minimum(c0, cap))
    np.testing.assert_array_equal(o["offsets"], offsets)
    np.testing.assert_array_equal(o["kept_pos"][: offsets[-1]], kpos)
    assert offsets[-1] <= budget
    if math.isfinite(tau):
        assert o["tau"] == np.float32(tau)
    np.testing.assert_allclose(o["dropped_uniform"], du, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(o["dropped_alloc"], da, rtol=1e-12, atol=1e-15)


def test_cap_that_truncates_nothing_is_the_plain_allocation():
    rng = np.random.default_rng(3)
    scores = np.exp(rng.normal(size=(6, 100)) * 1.5).astype(np.float32)
    a = oracle.contour_alloc(scores, 8, 240, 40)
    b = oracle.contour_alloc_capped(scores, 8, 240, 40, 100)
    for key in ("counts", "offsets", "kept_pos", "dropped_alloc", "dropped_uniform"):
        np.testing.assert_array_equal(a[key], b[key])


def test_cap_at_the_floor_keeps_only_the_floors():
    rng = np.random.default_rng(4)
    scores = np.exp(rng.normal(size=(5, 60))).astype(np.float32)
    o = oracle.contour_alloc_capped(scores, 16, 200, 40, 16)
    assert np.all(o["counts"] == 16)
    for h in range(5):
        np.testing.assert_array_equal(o["kept_pos"][o["offsets"][h]:o["offsets"][h + 1]], np.arange(44, 60))
    assert oracle.contour_alloc_capped(scores, 16, 200, 40, 15)["status"] == 1  # a cap below the floor


def test_ragged_store_compact_and_append_bytes():
    """Compaction into a store with room per cell, then decode-time appends,
    against slices written by hand; a cell without room takes nothing."""
    rng = np.random.default_rng(8)
    cells, T, d = 4, 30, 8
    K = rng.integers(0, 65535, size=(cells, T, d)).astype(np.uint16)
    V = rng.integers(0, 65535, size=(cells, T, d)).astype(np.uint16)
    scores = rng.random((cells, T)).astype(np.float32)
    o = oracle.contour_alloc(scores, 4, 40, 10)
    counts = np.diff(o["offsets"]).astype(np.int32)
    capacity = counts + np.array([3, 0, 5, 1], np.int32)
    capacity[3] = counts[3] - 1  # too small: the compaction skips this cell
    base = np.concatenate([[0], np.cumsum(capacity)[:-1]]).astype(np.int64) + 2  # two rows of slack first
    rows = int(base[-1] + capacity[-1])
    Ks = np.zeros((rows, d), np.uint16)
    Vs = np.zeros((rows, d), np.uint16)
    st = oracle.ragged_compact_to(K, V, o["offsets"], o["kept_pos"], base, capacity, Ks, Vs)
    np.testing.assert_array_equal(st, [0, 0, 0, 1])
    want_K = np.zeros_like(Ks)
    for h in range(3):
        a, b = o["offsets"][h], o["offsets"][h + 1]
        want_K[base[h]:base[h] + b - a] = K[h, o["kept_pos"][a:b]]
    np.testing.assert_array_equal(Ks, want_K)
    fill = counts.copy()
    fill[3] = 0
    for step in range(3):  # three decode steps of one row per cell
        nK = rng.integers(0, 65535, size=(cells, 1, d)).astype(np.uint16)
        nV = rng.integers(0, 65535, size=(cells, 1, d)).astype(np.uint16)
        before = fill.copy()
        st = oracle.ragged_append(Ks, Vs, base, capacity, fill, nK, nV)
        room = before + 1 <= capacity
        np.testing.assert_array_equal(st, (~room).astype(np.int32))
        np.testing.assert_array_equal(fill, before + room)
        for h in np.nonzero(room)[0]:
            np.testing.assert_array_equal(Ks[base[h] + before[h]], nK[h, 0])
            np.testing.assert_array_equal(Vs[base[h] + before[h]], nV[h, 0])
    assert Ks[0].sum() == 0 and Ks[1].sum() == 0  # the slack before the first cell is untouched
