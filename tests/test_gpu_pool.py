"""GPU parity for ES_pool (Definition 2.2): the exact best size-s subset of
the candidate set (top-mass set + the E dropped keys of largest single-key
error), through fw_pool_best_subset, against the fp64 oracle.

Sets must equal the oracle's unless the oracle records a near tie: between
its two best subsets (second gap within 1e-6 relative, or within the 1e-6 ||o||
floor that bounds the effect of the fp32 dense output), or at the pool
boundary (the E-th and (E+1)-th single-key errors within 1e-4 relative, where
the fp32 errors may admit the other key).  In those cases the CUDA set's gap
is compared with the oracle's es of that very set."""
import math

import numpy as np
import pytest

import oracle
import workloads
from tests.parity import ABS_FLOOR, NEAR_TIE, assert_close, np_, row_onorm
from tests.test_gpu_small import rows_batch

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

SCHED = [(4, 24), (8, 12), (16, 6), (32, 4)]  # (s, E): App. B's candidate-set schedule
POOL_NEAR = 1e-4


@pytest.fixture(scope="module")
def fw():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_25230_gb300 import fw as _fw

    return _fw


def row_host(H, r):
    """fp64 masses and values of row r of a HostRows batch."""
    g, i = divmod(int(r), H.R)
    n, d = int(H.n[g]), H.d
    off = int(H.logit_off[g]) + i * n
    l = H.logits[off:off + n].astype(np.float64)
    p = np.exp(l - l.max())
    p /= p.sum()
    V = H.v[int(H.v_off[g]):int(H.v_off[g]) + n * d]
    if H.v_dtype == 1:
        V = (V.astype(np.uint32) << 16).view(np.float32)
    return p, V.reshape(n, d).astype(np.float64)


def run_pool(fw, batch, E):
    rows = fw.rows_from_batch(batch)
    k = torch.as_tensor(np.asarray(batch.k)).cuda()
    top = fw.dense_and_topk_gap(rows, k)
    out = fw.pool_best_subset(rows, k, top, E=E)
    torch.cuda.synchronize()
    return rows, out


def check_pool(fw, batch, E, rows_index=None, out=None):
    """Compare (a sample of) rows with the oracle; returns the oracle dict."""
    if out is None:
        _, out = run_pool(fw, batch, E)
    H = oracle.HostRows(batch) if rows_index is None else rows_index[1]
    sel = slice(None) if rows_index is None else rows_index[0]
    o = oracle.pool_best_subset(H, E=E)
    assert o["call_status"] == 0
    on = row_onorm(oracle.dense_and_topk_gap(H)["o"])
    st = np_(out["row_status"])[sel]
    assert np.all(st == 0), st
    gi = np_(out["best_idx"])[sel]
    gg = np_(out["best_gap"])[sel]
    want = o["best_gap"].copy()
    k = np.asarray(H.k)
    for r in range(H.num_rows):
        for b in range(H.nb):
            s = int(k[r, b])
            mine = gi[r, b, :s]
            assert np.all(np.diff(mine) > 0) and np.all(gi[r, b, s:] == -1)
            theirs = o["best_idx"][r, b, :s]
            if np.array_equal(mine, theirs):
                continue
            near = (o["second_gap"][r, b] - o["best_gap"][r, b] <= NEAR_TIE * o["best_gap"][r, b] + ABS_FLOOR * on[r]
                    or o["pool_margin"][r, b] < POOL_NEAR)
            assert near, (r, b, mine, theirs, o["best_gap"][r, b], o["second_gap"][r, b], o["pool_margin"][r, b])
            p, Vr = row_host(H, r)
            mask = np.zeros(len(p), bool)
            mask[mine] = True
            want[r, b] = oracle.eval_instance(p, Vr, mask)["gap"]
    assert_close(gg, want, on, "ES_pool")
    assert_close(np_(out["topk_gap"])[sel], o["topk_gap"], on, "top-mass es")
    assert np.all(gg <= np_(out["topk_gap"])[sel] * (1 + 1e-6) + 1e-7 * on[:, None])
    return o, out


@pytest.mark.parametrize("n,d,v_dtype", [(33, 64, "f32"), (600, 128, "bf16"), (4097, 64, "f32"),
                                         (1000, 32, "bf16"), (300, 256, "f32")])
def test_pool_shapes(fw, n, d, v_dtype):
    rng = np.random.default_rng(n + d)
    rows = 10
    L = (rng.normal(size=(rows, n)) * rng.uniform(0.3, 4, size=(rows, 1))).astype(np.float32)
    L[:, 0] += 8
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    k = np.tile(np.array([s for s, _ in SCHED], np.int32), (rows, 1))
    check_pool(fw, rows_batch(L, V, k, v_dtype=v_dtype), [e for _, e in SCHED])


def test_pool_example_2_2(fw):
    # Example 2.2: p = (0.45, 0.45, 0.10), v = (-1, 1, 5) in one dimension,
    # s = 2; the pool is every key, ES_pool = ES(2) = 9/22 at {1, 3} (1-based),
    # the top-mass set {1, 2} has es 1/2.  Padded to 32 dims with zeros.
    p = np.array([0.45, 0.45, 0.10])
    L = np.log(p).astype(np.float32)[None, :]
    V = np.zeros((1, 3, 32), np.float32)
    V[0, :, 0] = [-1.0, 1.0, 5.0]
    _, out = run_pool(fw, rows_batch(L, V, [[2]]), [1])
    assert abs(float(np_(out["best_gap"])[0, 0]) - 9 / 22) <= 1e-6
    assert abs(float(np_(out["topk_gap"])[0, 0]) - 0.5) <= 1e-6
    np.testing.assert_array_equal(np_(out["best_idx"])[0, 0, :2], [0, 2])


def test_pool_of_every_key_is_the_exact_search(fw):
    # E >= n - s puts every key in the pool: ES_pool = ES(s), which the
    # separate exhaustive-search kernel (fw_best_subset) also computes
    rng = np.random.default_rng(7)
    rows, n, d = 24, 20, 64
    L = (rng.gumbel(size=(rows, n)) * rng.uniform(0.5, 3, size=(rows, 1))).astype(np.float32)
    L[:, 0] += 6
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    for s in (3, 5, 12):
        b = rows_batch(L, V, np.full((rows, 1), s))
        o, out = check_pool(fw, b, [n])
        rws = fw.rows_from_batch(b)
        bs = fw.best_subset(rws, torch.full((rows,), s, dtype=torch.int32, device="cuda"))
        torch.cuda.synchronize()
        on = row_onorm(oracle.dense_and_topk_gap(b)["o"])
        assert_close(np_(out["best_gap"])[:, 0], np_(bs["best_gap"]), on, "ES_pool vs ES")


@pytest.mark.parametrize("planted", [True, False])
def test_pool_hardness_instances(fw, planted):
    # App. A.2: uniform masses, integer points in one dimension, s = m/2.  A
    # planted balanced split gives ES = 0 exactly (many exact ties, settled by
    # the smallest colex rank); an odd total gives ES >= 2/m^2.
    m = 16
    if planted:
        w = np.array([3, 5, 2, 8, 1, 9, 4, 6, 7, 2, 5, 3, 8, 4, 6, 1], np.float32)
        w[-1] += w[::2].sum() - w[1::2].sum()  # even positions and odd positions balance
        assert w[::2].sum() == w[1::2].sum()
    else:
        w = np.array([3, 1, 4, 1, 5, 9, 2, 6, 5, 3, 5, 8, 9, 7, 9, 2], np.float32)
        assert int(w.sum()) % 2 == 1
    V = np.zeros((1, m, 32), np.float32)
    V[0, :, 0] = w
    b = rows_batch(np.zeros((1, m), np.float32), V, [[m // 2]])
    o, out = check_pool(fw, b, [m])
    g = float(np_(out["best_gap"])[0, 0])
    on = float(row_onorm(oracle.dense_and_topk_gap(b)["o"])[0])
    if planted:
        assert o["best_gap"][0, 0] <= 1e-12 * on and g <= ABS_FLOOR * on
    else:
        assert g >= 2.0 / m ** 2 * (1 - 1e-5)


def test_pool_degenerate_rows_take_the_fallback(fw):
    # every value equal: every subset has es = 0, so every one of the C(12, 4)
    # subsets is a re-scoring candidate and the warp's buffer overflows
    rng = np.random.default_rng(3)
    rows, n, d = 3, 40, 64
    L = rng.normal(size=(rows, n)).astype(np.float32)
    V = np.tile(rng.normal(size=(rows, 1, d)).astype(np.float32), (1, n, 1))
    V[2, 5:] += 1e-3 * rng.normal(size=(n - 5, d)).astype(np.float32)  # near-duplicates
    b = rows_batch(L, V, np.full((rows, 1), 4))
    _, out = run_pool(fw, b, [8])
    assert np.all(np_(out["n_cand"])[:2] == math.comb(12, 4))
    check_pool(fw, b, [8], out=out)


def test_pool_small_pools_and_budget_edges(fw):
    # E = 0 (the pool is the kept set: one subset), s = n, s = 1, s = 32
    rng = np.random.default_rng(9)
    rows, n, d = 6, 48, 64
    L = (rng.normal(size=(rows, n)) * 2).astype(np.float32)
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    k = np.tile(np.array([1, 7, 32, 20], np.int32), (rows, 1))
    check_pool(fw, rows_batch(L, V, k), [20, 0, 4, 5])
    k = np.full((rows, 1), 30, np.int32)
    check_pool(fw, rows_batch(L[:, :30].copy(), V[:, :30].copy(), k), [4])


def test_pool_refusals(fw):
    rng = np.random.default_rng(1)
    L = rng.normal(size=(3, 100)).astype(np.float32)
    V = rng.normal(size=(3, 100, 64)).astype(np.float32)
    k = np.array([[40], [5], [32]], np.int32)
    b = rows_batch(L, V, k)
    rws = fw.rows_from_batch(b)
    kd = torch.from_numpy(k).cuda()
    top = fw.dense_and_topk_gap(rws, kd)
    out = fw.pool_best_subset(rws, kd, top, E=[33])  # row 2: 32 + 33 > 64 pool keys
    torch.cuda.synchronize()
    np.testing.assert_array_equal(np_(out["row_status"]), [fw.FW_ERR_INVALID_ARG, 0, fw.FW_ERR_UNSUPPORTED])
    assert np.isnan(np_(out["best_gap"])[0, 0]) and np.isnan(np_(out["best_gap"])[2, 0])
    st, first = fw.sync_status(out["row_status"])
    assert (st, first) == (fw.FW_ERR_INVALID_ARG, 0)
    st, first = fw.sync_status(out["row_status"][1:2])
    assert (st, first) == (fw.FW_OK, -1)


def test_pool_mixed_profiles_sampled(fw):
    """Mixed-profile rows (GQA groups of 4 sharing bf16 V, n = 1,024 to 16,384)
    at the candidate-set schedule s = 4/8/16/32, E = 24/12/6/4; every row of a
    reduced batch against the oracle."""
    for b in workloads.mixed_profiles(seed=4, rows_scale=3e-4):
        nb = len(SCHED)
        R = b.num_rows
        b.k = np.tile(np.array([s for s, _ in SCHED], np.int32), (R, 1))
        b.nb = nb
        check_pool(fw, b, [e for _, e in SCHED])
