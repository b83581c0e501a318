"""GPU parity for the ContourKV variants (Sec. 4): the allocation with its
budget enforced per cell, compaction into ragged storage with room per cell,
and decode-time appends to it -- all bit-exact against the oracle."""
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


def check_capped(fw, scores, floor, budget, s, cap):
    sc = torch.as_tensor(np.asarray(scores, np.float32)).cuda() if not isinstance(scores, torch.Tensor) else scores
    g = fw.contour_alloc_capped(sc, floor=floor, total_budget=budget, uniform_s=s, cap=cap)
    torch.cuda.synchronize()
    o = oracle.contour_alloc_capped(sc.cpu().numpy(), floor, budget, s, cap)
    assert o["status"] == 0
    tot = int(o["offsets"][-1])
    np.testing.assert_array_equal(np_(g["counts"]), o["counts"])
    np.testing.assert_array_equal(np_(g["offsets"]), o["offsets"])
    np.testing.assert_array_equal(np_(g["kept_pos"])[:tot], o["kept_pos"][:tot])
    assert np_(g["tau"])[0] == np.float32(o["tau"])
    one = np.ones(len(o["counts"]))
    assert_close(np_(g["dropped_alloc"]), o["dropped_alloc"], one, "dropped_alloc")
    assert_close(np_(g["dropped_uniform"]), o["dropped_uniform"], one, "dropped_uniform")
    return g, o


@pytest.mark.parametrize("cells,T,floor,frac,cap", [(4, 100, 32, 0.5, 40), (8, 1000, 32, 1 / 8, 125),
                                                    (3, 31, 32, 1.0, 31), (16, 4096, 32, 1 / 8, 512),
                                                    (5, 300, 0, 0.1, 0), (7, 64, 8, 0.125, 8), (6, 2000, 16, 0.3, 5000)])
def test_capped_small(fw, cells, T, floor, frac, cap):
    cb = workloads.contour_cache(seed=cells + 30, cells=cells, T=T, with_kv=False, floor=floor, budget_frac=frac)
    budget = max(cells * min(floor, T), int(round(cells * T * frac)))
    check_capped(fw, cb.scores, floor, budget, budget // cells, max(cap, min(floor, T)))


# Cells split over several blocks: the cap's threshold found across slices,
# a cap at the floor (no non-floor entry kept), a cap above every count.
@pytest.mark.parametrize("cells,T,floor,frac,cap", [(3, 10000, 32, 0.3, 900), (4, 9001, 16, 0.2, 16),
                                                    (3, 9000, 0, 0.1, 0), (2, 8000, 8, 0.5, 100000)])
def test_capped_sliced(fw, cells, T, floor, frac, cap):
    cb = workloads.contour_cache(seed=cells + T + 1, cells=cells, T=T, with_kv=False, floor=floor, budget_frac=frac)
    budget = max(cells * min(floor, T), int(round(cells * T * frac)))
    check_capped(fw, cb.scores, floor, budget, budget // cells, max(cap, min(floor, T)))


def test_capped_sliced_ties(fw):
    rng = np.random.default_rng(6)
    s = (np.round(rng.lognormal(0, 1, size=(4, 9000)) * 4) / 4).astype(np.float32)
    check_capped(fw, s, 32, 4 * 1100, 1100, 900)
    check_capped(fw, np.ones((3, 9000), np.float32), 32, 3 * 2000, 2000, 1500)


def test_capped_ties(fw):
    rng = np.random.default_rng(4)
    s = np.round(rng.lognormal(0, 1, size=(12, 2000)) * 4) / 4  # equal scores at both thresholds
    check_capped(fw, s.astype(np.float32), 32, 12 * 250, 250, 200)
    check_capped(fw, np.ones((6, 500), np.float32), 32, 6 * 100, 100, 90)


def test_capped_full_scale_at_the_uniform_count(fw):
    """256 cells x 32,768 tokens, budget 1/8, every cell capped at the uniform
    per-cell count (4,096): the enforced mode of Sec. 4."""
    cb = workloads.contour_cache(seed=0, backend="torch", device="cuda", with_kv=False)
    g, o = check_capped(fw, cb.scores, cb.floor, cb.total_budget, cb.uniform_s, cb.uniform_s)
    assert np.all(o["counts"] <= cb.uniform_s) and o["offsets"][-1] < cb.total_budget


def test_ragged_store_and_decode_appends(fw):
    cells, T, d = 8, 900, 128
    cb = workloads.contour_cache(seed=12, cells=cells, T=T, d=d)
    sc = torch.as_tensor(cb.scores).cuda()
    g = fw.contour_alloc(sc, floor=32, total_budget=cb.total_budget, uniform_s=cb.uniform_s)
    counts = np_(g["counts"]).astype(np.int32)
    rng = np.random.default_rng(5)
    capacity = (counts + rng.integers(0, 4, size=cells)).astype(np.int32)
    capacity[2] = counts[2] - 1  # no room: compaction leaves the cell empty
    base = (np.concatenate([[0], np.cumsum(capacity)[:-1]]) + 16).astype(np.int64)
    rows = int(base[-1] + capacity[-1])
    K = torch.from_numpy(cb.K.view(np.int16)).cuda()
    V = torch.from_numpy(cb.V.view(np.int16)).cuda()
    Ks = torch.zeros(rows, d, dtype=torch.int16, device="cuda")
    Vs = torch.zeros_like(Ks)
    status = torch.empty(cells, dtype=torch.int32, device="cuda")
    bd, cd = torch.from_numpy(base).cuda(), torch.from_numpy(capacity).cuda()
    fw.ragged_compact_to(K, V, g["offsets"], g["kept_pos"], bd, cd, Ks, Vs, status)
    torch.cuda.synchronize()
    hK = np.zeros((rows, d), np.uint16)
    hV = np.zeros((rows, d), np.uint16)
    st = oracle.ragged_compact_to(cb.K, cb.V, np_(g["offsets"]), np_(g["kept_pos"]), base, capacity, hK, hV)
    # the oracle flags a cell without room with 1, the library with FW_ERR_WORKSPACE
    np.testing.assert_array_equal(np_(status), np.where(st != 0, fw.FW_ERR_WORKSPACE, 0))
    assert st[2] == 1 and st.sum() == 1
    np.testing.assert_array_equal(np_(Ks).view(np.uint16), hK)
    np.testing.assert_array_equal(np_(Vs).view(np.uint16), hV)
    fill = np.where(st == 0, counts, 0).astype(np.int32)
    fd = torch.from_numpy(fill.copy()).cuda()
    for m in (1, 1, 2, 1, 3):  # decode steps and a short prefill chunk
        nK = rng.integers(-32768, 32767, size=(cells, m, d)).astype(np.int16)
        nV = rng.integers(-32768, 32767, size=(cells, m, d)).astype(np.int16)
        fw.ragged_append(Ks, Vs, bd, cd, fd, torch.from_numpy(nK).cuda(), torch.from_numpy(nV).cuda(), status)
        st = oracle.ragged_append(hK, hV, base, capacity, fill, nK.view(np.uint16), nV.view(np.uint16))
        torch.cuda.synchronize()
        np.testing.assert_array_equal(np_(status), np.where(st != 0, fw.FW_ERR_WORKSPACE, 0))
        np.testing.assert_array_equal(np_(fd), fill)
    np.testing.assert_array_equal(np_(Ks).view(np.uint16), hK)
    np.testing.assert_array_equal(np_(Vs).view(np.uint16), hV)
