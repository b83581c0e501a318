"""The slice decomposition of the ContourKV allocation (Sec. 4), as a numpy
model checked against the oracle.

The device allocation splits each cell into S slices of consecutive
positions.  It counts, per slice, the non-floor keys above and equal to the
key that decides the cell (tau's, or the cap's when the cap keeps fewer), and
sums, per cell, the scores below each threshold.  From those it derives the
ties each cell takes, the counts and offsets, the dropped masses (the scores
below the threshold plus the ties not taken, each worth the threshold's
score), and for every slice the kept entries and ties of the cell's earlier
slices.  Its emit step then writes each slice's positions from there.

This model restates that arithmetic with numpy, for any S (the GPU tests
reach only the slice counts the library picks for their sizes), and checks
two things: the result equals the oracle's bit for bit, and every position a
slice writes lands inside its cell's range.  It shares no code with the CUDA
path; the thresholds come from sorting, not from a radix select."""
import numpy as np
import pytest

import oracle
import workloads


def score_key(x):
    # order key of a score >= 0 (-0 gets +0's key): the bits with the sign bit set
    x = np.where(x == 0, np.float32(0), x).astype(np.float32)
    return (x.view(np.uint32).astype(np.uint64) | 0x80000000)


def key_score(k):
    k = int(k)
    u = (k & 0x7fffffff) if (k & 0x80000000) else ((~k) & 0xffffffff)
    return float(np.array([u], np.uint32).view(np.float32)[0])


def kth(keys, k):
    """The key of rank k (1-based, descending) and the rank left among its equals."""
    t = int(np.sort(keys)[::-1][k - 1])
    return t, k - int((keys > t).sum())


def sliced_alloc(scores, floor, budget, us, cap, S):
    cells, T = scores.shape
    F = min(floor, T)
    nf = T - F
    K = budget - cells * F
    keys = score_key(scores)
    tk = kth(keys[:, :nf].ravel(), K)[0] if K > 0 else 0
    capnf = cap - F if cap >= 0 else -1
    cmode = 0 if (capnf < 0 or capnf >= nf) else (1 if capnf == 0 else 2)
    L = (((T + S - 1) // S) + 3) & ~3
    su = min(us, T)
    uT, urem, cT, crem = (np.zeros(cells, np.int64) for _ in range(4))
    for c in range(cells):
        if su > 0:
            uT[c], urem[c] = kth(keys[c], su)
        if cmode == 2:
            cT[c], crem[c] = kth(keys[c, :nf], capnf)

    def bounds(r):
        lo = min(T, r * L)
        return lo, min(T, lo + L)

    slot = {}
    for c in range(cells):
        for r in range(S):
            lo, hi = bounds(r)
            j = np.arange(lo, hi)
            k = keys[c, lo:hi]
            x = scores[c, lo:hi].astype(np.float64)
            m = j < nf
            d = dict(gt=0, eq=0, cgt=0, ceq=0, ueq=0, tot=x.sum())
            if K > 0:
                d.update(gt=int((m & (k > tk)).sum()), eq=int((m & (k == tk)).sum()), lt=x[m & (k < tk)].sum())
            else:
                d["lt"] = x[m].sum()
            if cmode == 2:
                d.update(cgt=int((m & (k > cT[c])).sum()), ceq=int((m & (k == cT[c])).sum()),
                         clt=x[m & (k < cT[c])].sum())
            else:
                d["clt"] = x[m].sum() if cmode == 1 else 0.0
            if su > 0:
                d.update(ueq=int((k == uT[c]).sum()), ult=x[k < uT[c]].sum())
            else:
                d["ult"] = x.sum()
            slot[c, r] = d
    ties_taken = K - sum(slot[c, r]["gt"] for c in range(cells) for r in range(S)) if K > 0 else 0
    ebefore = 0
    take, emode, counts = (np.zeros(cells, np.int64) for _ in range(3))
    da, du = np.zeros(cells), np.zeros(cells)
    for c in range(cells):
        def cs(f):
            return sum(slot[c, r][f] for r in range(S))
        gt, eq, ceq, ueq, tot = cs("gt"), cs("eq"), cs("ceq"), cs("ueq"), cs("tot")
        t = min(max(ties_taken - ebefore, 0), eq)
        ebefore += eq
        capped = cmode != 0 and gt + t > capnf
        cwant = int(crem[c]) if cmode == 2 else 0
        nonf = capnf if capped else gt + t
        take[c] = cwant if capped else t
        emode[c] = 2 if nonf == 0 else int(capped)
        counts[c] = F + nonf
        n = (ceq - cwant) if capped else (eq - t)
        thr = cT[c] if capped else tk
        dd = cs("clt" if capped else "lt") + (n * key_score(thr) if n > 0 else 0.0)
        da[c] = dd / tot if tot > 0 else 0.0
        n = ueq - int(urem[c])
        dd = cs("ult") + (n * key_score(uT[c]) if n > 0 else 0.0)
        du[c] = dd / tot if tot > 0 else 0.0
    offsets = np.concatenate([[0], np.cumsum(counts)])
    kept_pos = np.full(int(offsets[-1]), -1, np.int64)
    for c in range(cells):
        mode, want = emode[c], take[c]
        eT = cT[c] if mode == 1 else tk
        for r in range(S):
            tb = kb = 0  # ties and kept entries of the cell's earlier slices
            for q in range(r):
                sq = slot[c, q]
                e = 0 if mode == 2 else (sq["ceq"] if mode == 1 else sq["eq"])
                qlo, qhi = bounds(q)
                kb += max(0, qhi - max(qlo, nf))
                if mode != 2:
                    kb += (sq["cgt"] if mode == 1 else sq["gt"]) + min(max(want - tb, 0), e)
                tb += e
            lo, hi = bounds(r)
            w, rt = offsets[c] + kb, tb
            for j in range(lo, hi):
                kept = j >= nf
                if not kept and mode != 2:
                    if keys[c, j] > eT:
                        kept = True
                    elif keys[c, j] == eT:
                        kept = rt < want
                        rt += 1
                if kept:
                    assert offsets[c] <= w < offsets[c + 1], (c, r, j)
                    kept_pos[w] = j
                    w += 1
            if r == S - 1:
                assert w == offsets[c + 1]
    return dict(counts=counts, offsets=offsets, kept_pos=kept_pos, tau=key_score(tk) if K > 0 else np.inf,
                dropped_alloc=da, dropped_uniform=du)


def check(scores, floor, budget, us, cap, S):
    scores = np.asarray(scores, np.float32)
    g = sliced_alloc(scores, floor, budget, us, cap, S)
    o = (oracle.contour_alloc(scores, floor, budget, us) if cap < 0
         else oracle.contour_alloc_capped(scores, floor, budget, us, cap))
    assert o["status"] == 0
    tot = int(o["offsets"][-1])
    np.testing.assert_array_equal(g["counts"], o["counts"])
    np.testing.assert_array_equal(g["offsets"], o["offsets"])
    np.testing.assert_array_equal(g["kept_pos"][:tot], o["kept_pos"][:tot])
    assert np.float32(g["tau"]) == np.float32(o["tau"])
    np.testing.assert_allclose(g["dropped_alloc"], o["dropped_alloc"], rtol=1e-9, atol=1e-12)
    np.testing.assert_allclose(g["dropped_uniform"], o["dropped_uniform"], rtol=1e-9, atol=1e-12)


# (cells, T, floor, budget fraction, cap or -1, slices): ragged last slices,
# T not a multiple of 4, a floor spanning slices, a cap at the floor and one
# above every count, more slices than 4,096-position blocks would give
@pytest.mark.parametrize("cells,T,floor,frac,cap,S", [
    (3, 10000, 32, 1 / 8, -1, 3), (3, 10000, 32, 1 / 8, -1, 5), (5, 9999, 6000, 0.7, -1, 3),
    (2, 33333, 32, 1 / 8, -1, 8), (3, 10000, 32, 0.3, 900, 4), (4, 9001, 16, 0.2, 16, 3),
    (3, 9000, 0, 0.1, 0, 3), (2, 8000, 8, 0.5, 100000, 2), (3, 20, 32, 1.0, -1, 3), (3, 100, 8, 0.08, -1, 8)])
def test_sliced_allocation_matches_the_oracle(cells, T, floor, frac, cap, S):
    cb = workloads.contour_cache(seed=cells * 7 + T, cells=cells, T=T, with_kv=False, floor=floor, budget_frac=frac)
    budget = max(cells * min(floor, T), int(round(cells * T * frac)))
    check(cb.scores, floor, budget, budget // cells, cap if cap < 0 else max(cap, min(floor, T)), S)


@pytest.mark.parametrize("S", [1, 3, 8])
def test_sliced_allocation_ties_across_slices(S):
    rng = np.random.default_rng(1)
    s = (np.round(rng.lognormal(0, 1, size=(4, 9000)) * 4) / 4).astype(np.float32)
    ones = np.ones((3, 9000), np.float32)
    check(s, 32, 4 * 1100, 1100, -1, S)
    check(s, 32, 4 * 1100, 1100, 900, S)
    check(ones, 32, 3 * 2000, 2000, -1, S)  # every score equal
    check(ones, 32, 3 * 2000, 2000, 1500, S)
    check(s, 32, 4 * 32, 1100, -1, S)  # K = 0: the floors fill the budget
