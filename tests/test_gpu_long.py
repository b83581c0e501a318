"""GPU parity for long rows (n > 32): softmax statistics, radix top-k, P.V
products, forced-weight outputs, gap and dropped mass."""
import numpy as np
import pytest

import oracle
import workloads
from tests.parity import assert_close, np_, row_onorm
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
