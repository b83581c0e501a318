"""GPU parity for rows with n <= 32: top-k gap, swap rule, exact best subset.
Every test calls the CUDA path through the C ABI and compares with the fp64
oracle on the same seeded inputs."""
import math

import numpy as np
import pytest

import oracle
import workloads
from tests.parity import NEAR_TIE, assert_close, np_, row_onorm
from workloads import RowBatch

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def fw():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_25230_gb300 import fw as _fw

    return _fw


def rows_batch(L, V, k, v_dtype="f32", R=1):
    """L: [rows][n] logits; V: [groups][n][d]; k: [rows][nb]."""
    L = np.asarray(L, np.float32)
    rows, n = L.shape
    G = rows // R
    d = V.shape[2]
    if v_dtype == "bf16":
        vflat = workloads.f32_to_bf16_bits(np.asarray(V, np.float32)).ravel()
    else:
        vflat = np.asarray(V, np.float32).ravel()
    k = np.asarray(k, np.int32).reshape(rows, -1)
    return RowBatch(rows_per_group=R, d=d, n=np.full(G, n, np.int32), logits=L.ravel(),
                    logit_off=np.arange(G, dtype=np.int64) * R * n, v=vflat,
                    v_off=np.arange(G, dtype=np.int64) * n * d, v_dtype=v_dtype, k=k, nb=k.shape[1],
                    n_host=np.full(G, n, np.int32))


def check_gap(fw, batch):
    rows = fw.rows_from_batch(batch)
    k = torch.from_numpy(np.asarray(batch.k)).cuda()
    g = fw.dense_and_topk_gap(rows, k)
    torch.cuda.synchronize()
    o = oracle.dense_and_topk_gap(batch, words=(rows.max_n + 31) // 32)
    on = row_onorm(o["o"])
    assert np.all(np_(g["row_status"]) == 0)
    np.testing.assert_array_equal(np_(g["kept_bits"]).view(np.uint32), o["kept_bits"])
    assert_close(np_(g["gap"]), o["gap"], on, "gap")
    assert_close(np_(g["dropped"]), o["dropped"], on * 0 + 1, "dropped")  # dropped mass: floor 1e-6 absolute
    assert_close(np_(g["phi"]), o["phi"], on, "phi")
    assert_close(np_(g["o"]), o["o"], on, "o")
    assert_close(np_(g["o_kept"]), o["o_kept"], on, "o_kept")
    # the thresholds describe the same kept sets
    H = oracle.HostRows(batch)
    tk = np_(g["thr_key"]).view(np.uint32)
    ti = np_(g["thr_idx"])
    for r in range(min(H.num_rows, 64)):
        grp = r // H.R
        n = int(H.n[grp])
        l = H.logits[H.logit_off[grp] + (r % H.R) * n: H.logit_off[grp] + (r % H.R + 1) * n]
        u = np.where(l == 0, np.float32(0), l).view(np.uint32)
        key = np.where(u & 0x80000000, ~u, u | 0x80000000).astype(np.uint32)
        for b in range(H.nb):
            kept = (key > tk[r, b]) | ((key == tk[r, b]) & (np.arange(n) <= ti[r, b]))
            words = o["kept_bits"][r, b]
            want = np.array([(int(words[j >> 5]) >> (j & 31)) & 1 for j in range(n)], bool)
            np.testing.assert_array_equal(kept, want)
    return rows, k, g, o


def test_gap_exact_toy(fw):
    check_gap(fw, workloads.exact_toy(seed=0))


@pytest.mark.parametrize("n", [1, 2, 3, 17, 31, 32])
@pytest.mark.parametrize("d", [32, 64, 128, 256])
def test_gap_shapes_and_budgets(fw, n, d):
    rng = np.random.default_rng(n * 1000 + d)
    rows = 40
    L = (rng.normal(size=(rows, n)) * rng.uniform(0.2, 4, size=(rows, 1))).astype(np.float32)
    L[:, 0] += 5
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    ks = sorted({1, max(1, n - 1), n, max(1, n // 2)})
    k = np.tile(np.array(ks + [ks[-1]] * (4 - len(ks)), np.int32), (rows, 1))
    check_gap(fw, rows_batch(L, V, k))


def test_gap_ties_signed_zero_bf16_and_groups(fw):
    rng = np.random.default_rng(11)
    R, G, n, d = 4, 10, 24, 128
    L = np.round(rng.normal(size=(G * R, n)) * 2).astype(np.float32)  # many exact ties
    L[0, :] = 0.0
    L[1, ::2] = -0.0  # -0 and +0 tie, lower index first
    L[2, :] = 3.0     # all equal
    V = rng.normal(size=(G, n, d)).astype(np.float32)
    k = np.tile(np.array([1, 5, 12, 24], np.int32), (G * R, 1))
    check_gap(fw, rows_batch(L, V, k, v_dtype="bf16", R=R))


def test_gap_all_values_equal(fw):
    n, d, rows = 20, 64, 8
    rng = np.random.default_rng(12)
    L = rng.normal(size=(rows, n)).astype(np.float32)
    V = np.tile(rng.normal(size=(rows, 1, d)).astype(np.float32), (1, n, 1))
    rows_, k, g, o = check_gap(fw, rows_batch(L, V, np.full((rows, 1), 5)))
    assert np.all(np_(g["gap"]) <= 1e-6 * row_onorm(o["o"])[:, None])


def test_gap_nonfinite_row_is_flagged(fw):
    L = np.zeros((3, 8), np.float32)
    L[1, 3] = np.nan
    L[2, 0] = np.inf
    V = np.ones((3, 8, 32), np.float32)
    b = rows_batch(L, V, np.full((3, 1), 2))
    rows = fw.rows_from_batch(b)
    g = fw.dense_and_topk_gap(rows, torch.from_numpy(b.k).cuda())
    torch.cuda.synchronize()
    np.testing.assert_array_equal(np_(g["row_status"]), [0, 6, 6])


# ------------------------------------------------------------------ swap rule

def check_swap(fw, batch, E, max_swaps=16):
    rows = fw.rows_from_batch(batch)
    k = torch.from_numpy(np.asarray(batch.k)).cuda()
    top = fw.dense_and_topk_gap(rows, k)
    sw = fw.swap_refine(rows, k, top, E=E, max_swaps=max_swaps)
    torch.cuda.synchronize()
    o = oracle.swap_refine(batch, E=E, max_swaps=max_swaps)
    on = row_onorm(oracle.dense_and_topk_gap(batch)["o"])
    assert_close(np_(sw["topk_gap"]), o["topk_gap"], on, "swap topk_gap")
    exempt = (o["margin"] < NEAR_TIE) | (o["pool_margin"] < NEAR_TIE)
    ns, so, si = np_(sw["n_swaps"]), np_(sw["swap_out"]), np_(sw["swap_in"])
    strict = ~exempt
    np.testing.assert_array_equal(ns[strict], o["n_swaps"][strict])
    np.testing.assert_array_equal(so[strict], o["swap_out"][strict])
    np.testing.assert_array_equal(si[strict], o["swap_in"][strict])
    np.testing.assert_array_equal(np_(sw["capped"])[strict], o["capped"][strict])
    assert_close(np_(sw["refined_gap"]), o["refined_gap"], on, "refined_gap")
    return sw, o


def test_swap_exact_toy_all_keys(fw):
    b = workloads.exact_toy(seed=0)
    sw, o = check_swap(fw, b, E=20)
    assert np.all(o["refined_gap"] <= o["topk_gap"] * (1 + 1e-12))


@pytest.mark.parametrize("E", [0, 1, 4])
def test_swap_restricted_pool(fw, E):
    b = workloads.exact_toy(seed=1, rows=64, n=24, k=6, d=128)
    check_swap(fw, b, E=E)


def test_swap_budgets_and_cap(fw):
    rng = np.random.default_rng(21)
    rows, n, d = 48, 28, 64
    L = (rng.gumbel(size=(rows, n)) * rng.uniform(0.3, 3, size=(rows, 1))).astype(np.float32)
    L[:, 0] += 4
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    k = np.tile(np.array([2, 7, 14, 27], np.int32), (rows, 1))
    check_swap(fw, rows_batch(L, V, k), E=n, max_swaps=1)
    check_swap(fw, rows_batch(L, V, k), E=n, max_swaps=64)


# --------------------------------------------------------------- best subset

def check_best(fw, batch, sample=None):
    rows = fw.rows_from_batch(batch)
    k = torch.from_numpy(np.ascontiguousarray(np.asarray(batch.k)[:, 0])).cuda()
    bs = fw.best_subset(rows, k)
    torch.cuda.synchronize()
    H = oracle.HostRows(batch)
    o = oracle.best_subset(H)
    on = row_onorm(oracle.dense_and_topk_gap(H)["o"])
    assert np.all(np_(bs["row_status"]) == 0)
    assert_close(np_(bs["best_gap"]), o["best_gap"], on, "best_gap")
    assert_close(np_(bs["topk_gap"]), o["topk_gap"], on, "topk_gap")
    g1, g2 = o["best_gap"], o["second_gap"]
    tie = (g2 - g1) < NEAR_TIE * g1 + 1e-12 * on
    rk = np_(bs["best_rank"]).astype(np.uint64)
    np.testing.assert_array_equal(rk[~tie], o["best_rank"][~tie])
    idx = np_(bs["best_idx"])
    kk = np.asarray(batch.k)[:, 0]
    for r in range(len(kk)):
        members = idx[r, : kk[r]]
        assert np.all(np.diff(members) > 0)
        assert oracle.colex_rank(members) == int(rk[r])
        assert np.all(idx[r, kk[r]:] == -1)
    return bs, o


def test_best_exact_toy(fw):
    check_best(fw, workloads.exact_toy(seed=0))


def test_best_exact_enum_sample(fw):
    for b in workloads.exact_enum(seed=0, rows_scale=24 / 24192):
        check_best(fw, b)


@pytest.mark.parametrize("n,k", [(1, 1), (2, 1), (5, 5), (9, 3), (10, 4), (12, 11), (16, 8), (20, 1), (32, 2),
                                 (32, 3), (14, 9), (18, 10)])
def test_best_edges(fw, n, k):
    rng = np.random.default_rng(n * 100 + k)
    rows, d = 6, 64
    L = (rng.normal(size=(rows, n)) * 2).astype(np.float32)
    L[:, 0] += 3
    V = rng.normal(size=(rows, n, d)).astype(np.float32)
    check_best(fw, rows_batch(L, V, np.full((rows, 1), k)))


def test_best_degenerate_rows_take_the_exhaustive_path(fw):
    rng = np.random.default_rng(31)
    n, k, d = 16, 5, 64
    L = rng.normal(size=(4, n)).astype(np.float32)
    V = rng.normal(size=(4, n, d)).astype(np.float32)
    V[0] = V[0, :1]                     # all values equal: every subset has es = 0
    V[1, 1:] = V[1, 1]                  # all but one equal
    L[2] = 0.0                          # uniform masses
    check_best(fw, rows_batch(L, V, np.full((4, 1), k)))


@pytest.mark.parametrize("eps,d", [(1e-2, 64), (1e-3, 128), (1e-5, 64)])
def test_best_near_duplicate_values(fw, eps, d):
    # values scattered by eps around one point: many subsets within the fp32
    # bounds of the best, so rows overflow the candidate buffer and the
    # exhaustive path screens and re-scores them
    rng = np.random.default_rng(int(eps * 1e6) + d)
    rows, n, k = 8, 24, 6
    L = (rng.gumbel(size=(rows, n)) * rng.uniform(0.5, 2.0, size=(rows, 1))).astype(np.float32)
    base = rng.normal(size=(rows, 1, d))
    V = (base + eps * rng.normal(size=(rows, n, d))).astype(np.float32)
    check_best(fw, rows_batch(L, V, np.full((rows, 1), k)))


def test_best_hardness_instance(fw):
    # App. A.2 construction: d=1 padded to 32 dims with zeros, uniform masses, integer points
    m = 16
    w = np.array([3, 1, 4, 1, 5, 9, 2, 6, 5, 3, 5, 8, 9, 7, 9, 2], np.float32)  # sum 79 (odd) -> ES >= 2/m^2
    V = np.zeros((1, m, 32), np.float32)
    V[0, :, 0] = w
    bs, o = check_best(fw, rows_batch(np.zeros((1, m), np.float32), V, [[m // 2]]))
    assert np_(bs["best_gap"])[0] >= 2.0 / m ** 2 * (1 - 1e-5)


@pytest.mark.parametrize("kind", workloads.ADVERSARIAL_KINDS)
def test_best_adversarial_rows(fw, kind):
    """512 rows of each adversarial kind (flat rows, near-duplicate values,
    planted ES = 0 rows with exact ties) against the oracle, every row.  Where
    the oracle's best gap is exactly 0 (a planted row: every quantity is a short
    binary fraction, so the ties are exact on both sides) the rank must be the
    smallest colex rank among the tied subsets, the oracle's, with no near-tie
    exemption."""
    b = workloads.exact_adversarial(kind, rows=512, seed=0)
    bs, o = check_best(fw, b)
    zero = o["best_gap"] == 0.0
    if kind.startswith("planted"):
        assert zero.all()
        np.testing.assert_array_equal(np_(bs["best_rank"]).astype(np.uint64)[zero], o["best_rank"][zero])
        assert np.all(np_(bs["best_gap"])[zero] == 0.0)
    rows = fw.rows_from_batch(b)
    st = fw.best_subset_stats(rows, bs)
    print(f"{kind}: {st['rows_exhaustive']} of {rows.num_rows} rows on the exhaustive path, "
          f"{st['candidates']} candidates re-scored, {st['inner_leaves']} leaves visited")
    assert 0 <= st["rows_exhaustive"] <= rows.num_rows


def test_best_full_scale_sampled(fw):
    """The measured workload (168,192 rows, n=24, k=6) in one call per group:
    2,000 rows of every group (10,000 in all) against the oracle, properties on
    every row."""
    rng = np.random.default_rng(5)
    for b in workloads.exact_enum(seed=0, backend="torch", device="cuda"):
        rows = fw.rows_from_batch(b)
        k = b.k[:, 0].contiguous()
        top = fw.dense_and_topk_gap(rows, b.k, o_kept=False, kept_bits=False)
        bs = fw.best_subset(rows, k)
        torch.cuda.synchronize()
        best, tg = np_(bs["best_gap"]), np_(bs["topk_gap"])
        assert np.all(np_(bs["row_status"]) == 0)
        assert np.all(best <= tg * (1 + 1e-6))
        np.testing.assert_allclose(tg, np_(top["gap"])[:, 0], rtol=1e-5)
        assert np.all(np_(bs["best_rank"]) < math.comb(24, 6))
        pick = np.sort(rng.choice(rows.num_rows, 2000, replace=False))
        sub = _subset_rows(b, pick)
        o = oracle.best_subset(sub)
        on = row_onorm(oracle.dense_and_topk_gap(sub)["o"])
        assert_close(best[pick], o["best_gap"], on, "best_gap (sampled)")
        assert_close(tg[pick], o["topk_gap"], on, "topk_gap (sampled)")
        tie = (o["second_gap"] - o["best_gap"]) < NEAR_TIE * o["best_gap"]
        assert tie.mean() < 0.01
        np.testing.assert_array_equal(np_(bs["best_rank"])[pick][~tie].astype(np.uint64), o["best_rank"][~tie])
        idx = np_(bs["best_idx"])[pick]
        np.testing.assert_array_equal(idx[~tie], o["best_idx"][~tie])
        st = fw.best_subset_stats(rows, bs)
        print(f"group d={b.d}: {rows.num_rows} rows, {st['rows_exhaustive']} on the exhaustive path, "
              f"{st['candidates']} candidates, {st['inner_leaves']} leaves, {st['skipped']} skipped")
        del rows, top, bs, b
        torch.cuda.empty_cache()


def _subset_rows(b, pick):
    """Host copy of selected single-row groups of a torch RowBatch."""
    n, d = int(b.n_host[0]), b.d
    L = b.logits.view(-1, n)[torch.as_tensor(pick, device=b.logits.device)].cpu().numpy()
    V = b.v.view(-1, n, d)[torch.as_tensor(pick, device=b.v.device)].float().cpu().numpy()
    k = b.k[torch.as_tensor(pick, device=b.k.device)].cpu().numpy()
    return rows_batch(L, V, k)
