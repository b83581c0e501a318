"""GPU parity for the observation-window score (fw_window_score: TMA-fed
tcgen05 products of key tiles against the window queries) against the fp64
oracle, and ContourKV allocated on that score (Sec. 4's window-scored
variant).  Scores within 1e-4 relative (1e-6 of the cell's largest score as
the floor); the allocation on the CUDA scores bit-exact against the oracle's
allocation of the same scores."""
import math

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


def check(fw, Qb, Kb, pool=7, scale=None, cells_sel=None):
    """Qb, Kb: uint16 bf16 bits (numpy) or int16 device tensors."""
    Qd = torch.as_tensor(np.asarray(Qb).view(np.int16)).cuda() if isinstance(Qb, np.ndarray) else Qb
    Kd = torch.as_tensor(np.asarray(Kb).view(np.int16)).cuda() if isinstance(Kb, np.ndarray) else Kb
    d = Qd.shape[2]
    scale = 1 / math.sqrt(d) if scale is None else scale
    sc, st = fw.window_score(Qd, Kd, scale=scale, pool=pool)
    torch.cuda.synchronize()
    assert np.all(np_(st) == 0)
    sel = np.arange(Qd.shape[0]) if cells_sel is None else np.asarray(cells_sel)
    idx = torch.as_tensor(sel, device="cuda")
    qh = Qd[idx].cpu().numpy().view(np.uint16)
    kh = Kd[idx].cpu().numpy().view(np.uint16)
    want, _ = oracle.window_score(qh, kh, scale, pool)
    got = np_(sc)[sel]
    floor = want.max(axis=1)
    assert_close(got, want, floor, "window score")
    return sc, want


@pytest.mark.parametrize("cells,T,w,d", [(2, 300, 8, 64), (3, 1000, 32, 128), (1, 129, 32, 128), (4, 128, 1, 64),
                                         (2, 77, 16, 128), (5, 2048, 32, 64), (2, 40, 32, 128)])
def test_window_score_shapes(fw, cells, T, w, d):
    rng = np.random.default_rng(T * 7 + w)
    Q = workloads.f32_to_bf16_bits(rng.normal(size=(cells, w, d)).astype(np.float32))
    K = workloads.f32_to_bf16_bits((rng.normal(size=(cells, T, d)) * rng.uniform(0.5, 2.0)).astype(np.float32))
    check(fw, Q, K)


def test_window_score_pool_and_scale(fw):
    rng = np.random.default_rng(11)
    Q = workloads.f32_to_bf16_bits(rng.normal(size=(3, 12, 128)).astype(np.float32))
    K = workloads.f32_to_bf16_bits(rng.normal(size=(3, 700, 128)).astype(np.float32))
    check(fw, Q, K, pool=1)
    check(fw, Q, K, pool=15, scale=0.3)


def test_window_scored_contour_full_scale(fw):
    """The contour cache (256 cells x 32,768 tokens, d = 128, bf16 K) with a
    32-query window per cell: the score on eight cells against the oracle, then
    ContourKV on the CUDA scores at budget 1/8, bit-exact."""
    cb = workloads.contour_cache(seed=0, backend="torch", device="cuda")
    Qw = workloads.window_queries(seed=0, cells=cb.cells, w=32, d=cb.d, backend="torch", device="cuda")
    Kd = cb.K.view(torch.int16)
    sc, _ = check(fw, Qw.view(torch.int16), Kd, cells_sel=[0, 1, 77, 128, 200, 253, 254, 255])
    g = fw.contour_alloc(sc, floor=cb.floor, total_budget=cb.total_budget, uniform_s=cb.uniform_s)
    torch.cuda.synchronize()
    o = oracle.contour_alloc(np_(sc), cb.floor, cb.total_budget, cb.uniform_s)
    np.testing.assert_array_equal(np_(g["counts"]), o["counts"])
    np.testing.assert_array_equal(np_(g["kept_pos"]), o["kept_pos"])
