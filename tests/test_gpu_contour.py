"""GPU parity for ContourKV allocation and ragged compaction (bit-exact)."""
import numpy as np
import pytest

import oracle
import workloads
from tests.parity import assert_close, np_

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def fw():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_25230_gb300 import fw as _fw

    return _fw


def check(fw, scores, floor, budget, s):
    sc = torch.as_tensor(np.asarray(scores, np.float32)).cuda() if not isinstance(scores, torch.Tensor) else scores
    g = fw.contour_alloc(sc, floor=floor, total_budget=budget, uniform_s=s)
    torch.cuda.synchronize()
    o = oracle.contour_alloc(sc.cpu().numpy(), floor, budget, s)
    assert o["status"] == 0
    np.testing.assert_array_equal(np_(g["counts"]), o["counts"])
    np.testing.assert_array_equal(np_(g["offsets"]), o["offsets"])
    np.testing.assert_array_equal(np_(g["kept_pos"]), o["kept_pos"])
    assert np_(g["tau"])[0] == np.float32(o["tau"])
    one = np.ones(len(o["counts"]))
    assert_close(np_(g["dropped_alloc"]), o["dropped_alloc"], one, "dropped_alloc")
    assert_close(np_(g["dropped_uniform"]), o["dropped_uniform"], one, "dropped_uniform")
    return g, o


@pytest.mark.parametrize("cells,T,floor,frac", [(4, 100, 32, 0.5), (8, 1000, 32, 1 / 8), (3, 31, 32, 1.0),
                                                 (16, 4096, 32, 1 / 8), (5, 300, 0, 0.1), (7, 64, 8, 0.125)])
def test_contour_small(fw, cells, T, floor, frac):
    cb = workloads.contour_cache(seed=cells, cells=cells, T=T, with_kv=False, floor=floor, budget_frac=frac)
    budget = max(cells * min(floor, T), int(round(cells * T * frac)))
    check(fw, cb.scores, floor, budget, budget // cells)


def test_contour_ties(fw):
    rng = np.random.default_rng(1)
    s = np.round(rng.lognormal(0, 1, size=(12, 2000)) * 4) / 4  # many equal scores across cells
    check(fw, s.astype(np.float32), 32, 12 * 250, 250)
    check(fw, np.ones((6, 500), np.float32), 32, 6 * 100, 100)  # every score equal


# Cells long enough to be split over several blocks (slices of >= 4,096
# positions, up to 8 per cell): ragged last slices, T not a multiple of 4 (the
# scalar path), a floor spanning slices, ties at tau across slice boundaries,
# every score equal, and K = 0 (the floors fill the budget).
@pytest.mark.parametrize("cells,T,floor,frac", [(3, 10000, 32, 1 / 8), (2, 33333, 32, 1 / 8),
                                                 (5, 9999, 6000, 0.7), (2, 65536, 32, 1 / 16)])
def test_contour_sliced(fw, cells, T, floor, frac):
    cb = workloads.contour_cache(seed=cells + T, cells=cells, T=T, with_kv=False, floor=floor, budget_frac=frac)
    budget = max(cells * min(floor, T), int(round(cells * T * frac)))
    check(fw, cb.scores, floor, budget, budget // cells)


def test_contour_sliced_ties(fw):
    rng = np.random.default_rng(5)
    s = (np.round(rng.lognormal(0, 1, size=(4, 9000)) * 4) / 4).astype(np.float32)
    check(fw, s, 32, 4 * 1100, 1100)
    check(fw, np.ones((3, 9000), np.float32), 32, 3 * 2000, 2000)
    check(fw, s, 32, 4 * 32, 1100)  # K = 0


def test_compaction_small(fw):
    rng = np.random.default_rng(2)
    cells, T, d = 6, 700, 128
    cb = workloads.contour_cache(seed=9, cells=cells, T=T, d=d)
    g = fw.contour_alloc(torch.as_tensor(cb.scores).cuda(), floor=32, total_budget=cb.total_budget,
                         uniform_s=cb.uniform_s)
    K = torch.from_numpy(cb.K.view(np.int16)).cuda()
    V = torch.from_numpy(cb.V.view(np.int16)).cuda()
    Ko, Vo = fw.ragged_compact(K, V, g["offsets"], g["kept_pos"], cb.total_budget)
    torch.cuda.synchronize()
    o = oracle.contour_alloc(cb.scores, 32, cb.total_budget, cb.uniform_s)
    rk, rv = oracle.ragged_compact(cb.K, cb.V, o["offsets"], o["kept_pos"])
    np.testing.assert_array_equal(np_(Ko).view(np.uint16), rk)
    np.testing.assert_array_equal(np_(Vo).view(np.uint16), rv)
    assert rng is not None


def test_contour_and_compaction_full_scale(fw):
    """32 layers x 8 heads = 256 cells x 32,768 tokens, d=128 bf16, budget 1/8."""
    cb = workloads.contour_cache(seed=0, backend="torch", device="cuda")
    g, o = check(fw, cb.scores, cb.floor, cb.total_budget, cb.uniform_s)
    K = cb.K.view(torch.int16)
    V = cb.V.view(torch.int16)
    Ko, Vo = fw.ragged_compact(K, V, g["offsets"], g["kept_pos"], cb.total_budget)
    torch.cuda.synchronize()
    rk, rv = oracle.ragged_compact(K.cpu().numpy().view(np.uint16), V.cpu().numpy().view(np.uint16),
                                   o["offsets"], o["kept_pos"])
    assert np.array_equal(np_(Ko).view(np.uint16), rk)
    assert np.array_equal(np_(Vo).view(np.uint16), rv)
