"""GPU parity for long rows (n > 32): softmax statistics, radix top-k, P.V
products, forced-weight outputs, gap and dropped mass."""
import numpy as np
import pytest

import oracle
import workloads
from tests.parity import assert_close, close, np_, row_onorm
from tests.test_gpu_small import rows_batch

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def fw():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_25230_gb300 import fw as _fw

    return _fw


def compare(fw, batch, rows=None, g=None, pick=None):
    """Run (unless given) and compare every row, or the rows in `pick`."""
    if rows is None:
        rows = fw.rows_from_batch(batch)
        g = fw.dense_and_topk_gap(rows, torch.as_tensor(np.asarray(batch.k) if not hasattr(batch.k, "cuda")
                                                          else batch.k).cuda())
        torch.cuda.synchronize()
    H = oracle.HostRows(batch) if pick is None else pick.H
    o = oracle.dense_and_topk_gap(H, words=(rows.max_n + 31) // 32)
    sel = slice(None) if pick is None else pick.rows_index
    on = row_onorm(o["o"])
    assert np.all(np_(g["row_status"])[sel] == 0)
    np.testing.assert_array_equal(np_(g["kept_bits"])[sel].view(np.uint32), o["kept_bits"])
    assert_close(np_(g["gap"])[sel], o["gap"], on, "gap")
    assert_close(np_(g["dropped"])[sel], o["dropped"], np.ones_like(on), "dropped")
    assert_close(np_(g["phi"])[sel], o["phi"], on, "phi")
    assert_close(np_(g["o"])[sel], o["o"], on, "o")
    assert_close(np_(g["o_kept"])[sel], o["o_kept"], on, "o_kept")
    return rows, g, o


@pytest.mark.parametrize("n", [33, 100, 1000, 4097])
def test_long_shapes(fw, n):
    rng = np.random.default_rng(n)
    rows, d = 12, 64
    L = (rng.normal(size=(rows, n)) * rng.uniform(0.3, 4, size=(rows, 1))).astype(np.float32)
    L[:, 0] += 8
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    k = np.tile(np.array([1, max(1, n // 16), n // 4, n], np.int32), (rows, 1))
    compare(fw, rows_batch(L, V, k))


def test_long_rows_reduced(fw):
    # the long-row workload's structure at a size the oracle checks in seconds
    b = workloads.long_rows(seed=0, heads=2, rows_per_head=12, n=4096)
    compare(fw, b)


def test_long_ties_and_groups(fw):
    rng = np.random.default_rng(3)
    R, G, n, d = 8, 3, 777, 128
    L = np.round(rng.normal(size=(G * R, n)) * 1.5).astype(np.float32)  # heavy ties
    L[0] = 1.0                         # one row all equal
    L[1, ::3] = -0.0
    L[1, 1::3] = 0.0
    V = rng.normal(size=(G, n, d)).astype(np.float32)
    k = np.tile(np.array([3, 64, 200], np.int32), (G * R, 1))
    compare(fw, rows_batch(L, V, k, v_dtype="bf16", R=R))


@pytest.mark.parametrize("nb,d", [(1, 64), (2, 128), (3, 64), (4, 128)])
def test_long_bf16_band_counts(fw, nb, d):
    # bf16 values take the tensor-core P.V; nb + 1 bands per row set the tile
    # height (32 rows, or 25 for five bands) and 70 rows per group leave a
    # partial tile; n = 1000 leaves a partial 64-key stage
    rng = np.random.default_rng(10 * nb + d)
    R, G, n = 70, 2, 1000
    L = (rng.normal(size=(G * R, n)) * rng.uniform(0.5, 3.0, size=(G * R, 1))).astype(np.float32)
    L[:, 0] += 5.0
    V = rng.normal(size=(G, n, d)).astype(np.float32)
    ks = [7, 100, 333, 999][:nb]
    k = np.tile(np.array(ks, np.int32), (G * R, 1))
    compare(fw, rows_batch(L, V, k, v_dtype="bf16", R=R))


@pytest.mark.parametrize("R,nb,d", [(1, 1, 64), (3, 2, 128), (4, 1, 64), (4, 4, 128), (5, 3, 64), (8, 4, 128),
                                    (8, 2, 64), (2, 3, 128)])
def test_long_bf16_small_groups(fw, R, nb, d):
    # groups of at most 8 rows take the transposed P.V (value dims on the
    # MMA's M, (band, row) pairs on N); n = 1000 leaves a partial 64-key stage,
    # n = 1001 also sends the logits through 4-byte copies
    for n in (1000, 1001, 4096):
        rng = np.random.default_rng(100 * R + 10 * nb + d + n)
        G = 5
        L = (rng.normal(size=(G * R, n)) * rng.uniform(0.3, 3.0, size=(G * R, 1))).astype(np.float32)
        L[:, 0] += 5.0
        V = rng.normal(size=(G, n, d)).astype(np.float32)
        ks = [7, 100, 333, n - 1][:nb]
        k = np.tile(np.array(ks, np.int32), (G * R, 1))
        compare(fw, rows_batch(L, V, k, v_dtype="bf16", R=R))


def test_mixed_profiles_reduced(fw):
    for b in workloads.mixed_profiles(seed=0, rows_scale=2e-3):
        compare(fw, b)


class _Pick:
    """Host copy of a few rows of a device RowBatch, with their row indices."""

    def __init__(self, b, rows_index):
        self.rows_index = np.asarray(rows_index)
        R = b.rows_per_group
        n = int(b.n_host[0])
        d = b.d
        groups = self.rows_index // R
        L = b.logits.view(-1, n)[torch.as_tensor(self.rows_index, device=b.logits.device)].cpu().numpy()
        Vg = b.v.view(-1, n, d)[torch.as_tensor(groups, device=b.v.device)].view(torch.int16).cpu().numpy()
        k = b.k[torch.as_tensor(self.rows_index, device=b.k.device)].cpu().numpy()
        batch = workloads.RowBatch(rows_per_group=1, d=d, n=np.full(len(groups), n, np.int32), logits=L.ravel(),
                                   logit_off=np.arange(len(groups), dtype=np.int64) * n,
                                   v=Vg.view(np.uint16).ravel(),
                                   v_off=np.arange(len(groups), dtype=np.int64) * n * d, v_dtype="bf16", k=k,
                                   nb=k.shape[1], n_host=np.full(len(groups), n, np.int32))
        self.H = oracle.HostRows(batch)
        for a in ("R", "d", "n", "logits", "logit_off", "v", "v_off", "v_dtype", "k", "nb", "num_rows", "max_n",
                  "c"):
            setattr(self, a, getattr(self.H, a))


def test_long_rows_full_scale_sampled(fw):
    """8 KV heads x 512 rows x 32,768 keys, three budgets, as measured."""
    b = workloads.long_rows(seed=0, backend="torch", device="cuda")
    rows = fw.rows_from_batch(b)
    g = fw.dense_and_topk_gap(rows, b.k)
    torch.cuda.synchronize()
    pick = np.sort(np.random.default_rng(0).choice(rows.num_rows, 6, replace=False))
    compare(fw, None, rows=rows, g=g, pick=_Pick(b, pick))
    # properties on every row
    gap, dr = np_(g["gap"]), np_(g["dropped"])
    assert np.all(np_(g["row_status"]) == 0)
    assert np.all(np.diff(dr, axis=1) <= 1e-7)  # nested budgets drop less mass
    assert np.all(np.isfinite(gap))


# ------------------------------------------------------------ swap rule, long rows

def check_swap_long(fw, batch, E=32, max_swaps=16):
    from tests.parity import NEAR_TIE

    rows = fw.rows_from_batch(batch)
    k = torch.as_tensor(np.asarray(batch.k)).cuda()
    top = fw.dense_and_topk_gap(rows, k)
    sw = fw.swap_refine(rows, k, top, E=E, max_swaps=max_swaps)
    torch.cuda.synchronize()
    o = oracle.swap_refine(batch, E=E, max_swaps=max_swaps)
    on = row_onorm(oracle.dense_and_topk_gap(batch)["o"])
    assert_close(np_(sw["topk_gap"]), o["topk_gap"], on, "swap topk_gap")
    exempt = (o["margin"] < NEAR_TIE) | (o["pool_margin"] < NEAR_TIE)
    strict = ~exempt
    assert strict.mean() > 0.5  # most decisions are not near-ties
    np.testing.assert_array_equal(np_(sw["n_swaps"])[strict], o["n_swaps"][strict])
    np.testing.assert_array_equal(np_(sw["swap_out"])[strict], o["swap_out"][strict])
    np.testing.assert_array_equal(np_(sw["swap_in"])[strict], o["swap_in"][strict])
    np.testing.assert_array_equal(np_(sw["capped"])[strict], o["capped"][strict])
    assert_close(np_(sw["refined_gap"]), o["refined_gap"], on, "refined_gap")
    assert np.all(np_(sw["refined_gap"]) <= np_(sw["topk_gap"]) * (1 + 1e-6))
    return sw, o


def test_swap_long_rows_reduced(fw):
    b = workloads.long_rows(seed=1, heads=2, rows_per_head=6, n=2048)
    check_swap_long(fw, b)


@pytest.mark.parametrize("n,E", [(40, 32), (300, 8), (1000, 32)])
def test_swap_long_shapes(fw, n, E):
    rng = np.random.default_rng(n + E)
    rows, d = 8, 64
    L = (rng.normal(size=(rows, n)) * rng.uniform(0.3, 3, size=(rows, 1))).astype(np.float32)
    L[:, 0] += 6
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    k = np.tile(np.array([1, max(1, n // 8), n // 2], np.int32), (rows, 1))
    check_swap_long(fw, rows_batch(L, V, k), E=E, max_swaps=8)


def test_swap_mixed_profiles_reduced(fw):
    for b in workloads.mixed_profiles(seed=2, rows_scale=6e-4,
                                      profiles=(("A", 36864, 64, 1024), ("B", 24192, 128, 4096))):
        check_swap_long(fw, b)


class _PickRagged:
    """Host copy of a few rows of a device RowBatch whose groups differ in n."""

    def __init__(self, b, rows_index):
        self.rows_index = np.asarray(rows_index)
        R = b.rows_per_group
        d = b.d
        n_host = np.asarray(b.n_host)
        lo = b.logit_off.cpu().numpy() if hasattr(b.logit_off, "cpu") else np.asarray(b.logit_off)
        vo = b.v_off.cpu().numpy() if hasattr(b.v_off, "cpu") else np.asarray(b.v_off)
        Ls, Vs, ns = [], [], []
        for r in self.rows_index:
            g = int(r) // R
            n = int(n_host[g])
            off = int(lo[g]) + (int(r) - g * R) * n
            Ls.append(b.logits[off:off + n].cpu().numpy())
            Vs.append(b.v[int(vo[g]):int(vo[g]) + n * d].view(torch.int16).cpu().numpy().view(np.uint16))
            ns.append(n)
        ns = np.asarray(ns, np.int32)
        k = b.k[torch.as_tensor(self.rows_index, device=b.k.device)].cpu().numpy()
        batch = workloads.RowBatch(rows_per_group=1, d=d, n=ns, logits=np.concatenate(Ls),
                                   logit_off=np.concatenate([[0], np.cumsum(ns)[:-1]]).astype(np.int64),
                                   v=np.concatenate(Vs),
                                   v_off=np.concatenate([[0], np.cumsum(ns.astype(np.int64) * d)[:-1]]).astype(np.int64),
                                   v_dtype="bf16", k=k, nb=k.shape[1], n_host=ns)
        self.H = oracle.HostRows(batch)


POOL_NEAR = 1e-4  # pool-boundary margin below which the fp32 single-key errors may admit the other key
CHAIN_BAND = 1e-6  # near-tie band of one round's choice, relative to that round's es


def _check_chain(H, r, b, E, n_sw, s_out, s_in, capped, refined, onr, kept_bits):
    """Replays one swap chain of the CUDA path with the oracle's full round
    scores (orc_swap_scores: es of every kept x pool option, fp64).  Each taken
    swap must remove a kept key and add a pool key outside the set, must lower
    es (within the band), and must be within CHAIN_BAND of that round's best
    option; the final set must admit no pool swap that lowers es by more than
    the band, and its es must be the refined gap the CUDA path reports.  Where
    the pool boundary itself is a near tie, the added keys may come from the
    CUDA path's own pool (one key either side of the boundary), and the final
    local-optimality test is over the union of both pools' candidates."""
    k = int(H.k[r, b])
    pool, pm = oracle.candidate_set(H, r, k, E)
    near_pool = pm < POOL_NEAR
    n = int(H.n[r // H.R])
    A = np.array([(int(kept_bits[j >> 5]) >> (j & 31)) & 1 for j in range(n)], bool)
    assert A.sum() == k
    extra = set()
    for t in range(int(n_sw)):
        i, j = int(s_out[t]), int(s_in[t])
        assert A[i] and not A[j], (r, b, t, i, j)
        if j not in set(pool.tolist()):
            assert near_pool, (r, b, t, j)
            extra.add(j)
        add = np.array(sorted(set(x for x in pool.tolist() if not A[x]) | {x for x in extra if not A[x]}), np.int32)
        scores, cur = oracle.swap_scores(H, r, A, add)
        kept = np.flatnonzero(A)
        taken = scores[np.searchsorted(kept, i), np.searchsorted(add, j)]
        band = CHAIN_BAND * cur + 1e-7 * onr
        assert taken <= scores.min() + band, (r, b, t, taken, scores.min(), cur)
        assert taken < cur + band, (r, b, t, taken, cur)
        A[i], A[j] = False, True
    add = np.array(sorted(set(x for x in pool.tolist() if not A[x]) | {x for x in extra if not A[x]}), np.int32)
    scores, cur = oracle.swap_scores(H, r, A, add)
    if scores.size and not capped and not near_pool:
        assert scores.min() >= cur - (CHAIN_BAND * cur + 1e-7 * onr), (r, b, scores.min(), cur)
    assert abs(refined - cur) <= 1e-4 * cur + 1e-6 * onr, (r, b, refined, cur)


def _compare_swap(sw, o, sel, on, H, E):
    """Swap outputs of the sampled rows against the oracle.  Over ~30 rounds of
    up to 8,192 x 32 candidate pairs, many (row, budget) chains contain a
    decision closer than 1e-6 relative (the oracle's `margin`), after which the
    greedy paths may part.  Chains without such a decision must equal the
    oracle's exactly; every chain, with or without, is replayed round by round
    against the oracle's full scores of that round (_check_chain)."""
    from tests.parity import NEAR_TIE

    exempt = (o["margin"] < NEAR_TIE) | (o["pool_margin"] < NEAR_TIE)
    strict = ~exempt
    assert_close(np_(sw["topk_gap"])[sel], o["topk_gap"], on, "swap topk_gap")
    for key in ("n_swaps", "capped", "swap_out", "swap_in"):
        np.testing.assert_array_equal(np_(sw[key])[sel][strict], o[key][strict])
    rg = np_(sw["refined_gap"])[sel]
    ok = close(rg, o["refined_gap"], on)
    assert np.all(ok[strict]), "refined_gap differs on a chain without near-ties"
    assert np.all(rg <= np_(sw["topk_gap"])[sel] * (1 + 1e-6))
    kb = oracle.dense_and_topk_gap(H)["kept_bits"]
    ns, so, si, cp = (np_(sw[x])[sel] for x in ("n_swaps", "swap_out", "swap_in", "capped"))
    for r in range(H.num_rows):
        for b in range(H.nb):
            _check_chain(H, r, b, E, ns[r, b], so[r, b], si[r, b], cp[r, b], float(rg[r, b]), float(on[r]),
                         kb[r, b])
    return int(strict.sum())


def test_swap_long_rows_full_scale_sampled(fw):
    """The swap rule on the measured long-row workload (4,096 rows x 32,768
    keys, budgets 2,048 / 4,096 / 8,192, E = 32, at most 64 swaps), as timed;
    four rows re-run by the oracle, properties on every row."""
    b = workloads.long_rows(seed=0, backend="torch", device="cuda")
    rows = fw.rows_from_batch(b)
    g = fw.dense_and_topk_gap(rows, b.k)
    sw = fw.swap_refine(rows, b.k, g, E=32, max_swaps=64)
    torch.cuda.synchronize()
    pick = _Pick(b, np.sort(np.random.default_rng(1).choice(rows.num_rows, 4, replace=False)))
    o = oracle.swap_refine(pick.H, E=32, max_swaps=64)
    on = row_onorm(oracle.dense_and_topk_gap(pick.H)["o"])
    _compare_swap(sw, o, pick.rows_index, on, pick.H, 32)
    # on every row: finite, never worse than the top-k set, never capped
    rg, tg = np_(sw["refined_gap"]), np_(sw["topk_gap"])
    assert np.all(np.isfinite(rg)) and np.all(rg <= tg * (1 + 1e-6))
    assert np.all(np_(sw["capped"]) == 0)


def test_mixed_profiles_full_scale_sampled(fw):
    """The mixed-profile sweep at full size (168,192 rows in GQA groups of 4,
    n from 1,024 to 16,384, bf16 V), profile by profile: gap and swap rule on
    every row, three rows of each profile re-run by the oracle, properties on
    every row."""
    rng = np.random.default_rng(5)
    # one profile at a time keeps the device footprint of generation below
    # ~100 GB (profile E: 18,432 rows x 16,384 keys, 19 GB of bf16 values)
    for prof in workloads.MIXED_PROFILES:
        b = workloads.mixed_profiles(seed=0, backend="torch", device="cuda", profiles=(prof,))[0]
        rows = fw.rows_from_batch(b)
        g = fw.dense_and_topk_gap(rows, b.k)
        sw = fw.swap_refine(rows, b.k, g, E=32, max_swaps=64)
        torch.cuda.synchronize()
        assert np.all(np_(g["row_status"]) == 0)
        gap, dr = np_(g["gap"]), np_(g["dropped"])
        assert np.all(np.isfinite(gap)) and np.all((dr >= 0) & (dr <= 1 + 1e-6))
        rg, tg = np_(sw["refined_gap"]), np_(sw["topk_gap"])
        assert np.all(np.isfinite(rg)) and np.all(rg <= tg * (1 + 1e-6))
        # one row from the first, a middle and the last group
        G = rows.num_rows // b.rows_per_group
        groups = [0, G // 2, G - 1]
        sel = np.array([gi * b.rows_per_group + int(rng.integers(b.rows_per_group)) for gi in groups])
        pick = _PickRagged(b, sel)
        og = oracle.dense_and_topk_gap(pick.H)
        on = row_onorm(og["o"])
        assert_close(gap[sel], og["gap"], on, "gap")
        assert_close(dr[sel], og["dropped"], np.ones_like(on), "dropped")
        assert_close(np_(g["o"])[sel], og["o"], on, "o")
        o = oracle.swap_refine(pick.H, E=32, max_swaps=64)
        _compare_swap(sw, o, sel, on, pick.H, 32)
        del rows, g, sw, b
        torch.cuda.empty_cache()
