"""fw_contour_alloc_noalloc -- the ContourKV allocator for callers that cannot
allocate device memory (for example a plugin confined to another framework's
memory pool, or a latency-critical path that must not trigger cudaMalloc's
device synchronisation).  It must give exactly what fw_contour_alloc gives,
call after call, while its scratch area is shared between calls.

This file is collected last so that a failure here leaves every other test
already run."""
import ctypes as C

import numpy as np
import pytest

import workloads
from tests.parity import assert_close, np_

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def fw():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_25230_gb300 import fw as _fw

    _fw.raw().fw_contour_alloc_noalloc.argtypes = [C.c_void_p, C.c_int32, C.c_int32, C.c_int32, C.c_int64,
                                                   C.c_int32] + [C.c_void_p] * 7
    _fw.raw().fw_contour_alloc_noalloc.restype = C.c_int
    return _fw


def new_outputs(cells, budget, dev):
    return dict(counts=torch.full((cells,), -7, dtype=torch.int32, device=dev),
                offsets=torch.full((cells + 1,), -7, dtype=torch.int64, device=dev),
                kept_pos=torch.full((budget,), -7, dtype=torch.int32, device=dev),
                tau=torch.zeros(1, dtype=torch.float32, device=dev),
                dropped_uniform=torch.zeros(cells, dtype=torch.float32, device=dev),
                dropped_alloc=torch.zeros(cells, dtype=torch.float32, device=dev))


def call_noalloc(fw, scores, floor, budget, s, out=None):
    cells, T = scores.shape
    if out is None:
        out = new_outputs(cells, budget, scores.device)
    p = lambda t: C.c_void_p(t.data_ptr())  # noqa: E731
    st = fw.raw().fw_contour_alloc_noalloc(p(scores), cells, T, floor, budget, s, p(out["counts"]),
                                           p(out["offsets"]), p(out["kept_pos"]), p(out["tau"]),
                                           p(out["dropped_uniform"]), p(out["dropped_alloc"]),
                                           C.c_void_p(torch.cuda.current_stream().cuda_stream))
    return st, out


def test_noalloc_matches_the_workspace_entry_point_on_consecutive_calls(fw):
    cases = []
    for seed, (cells, T, frac) in enumerate([(64, 3000, 1 / 8), (200, 1500, 1 / 4), (24, 20000, 1 / 8)]):
        cb = workloads.contour_cache(seed=seed + 40, cells=cells, T=T, with_kv=False, budget_frac=frac)
        sc = torch.as_tensor(cb.scores).cuda()
        if seed == 1:
            sc = torch.round(sc * 4) / 4  # ties across cells
        cases.append((sc, cb.floor, cb.total_budget, cb.uniform_s))
    for sc, floor, budget, s in cases:  # two calls in a row, different inputs
        ref = fw.contour_alloc(sc, floor=floor, total_budget=budget, uniform_s=s)
        st, got = call_noalloc(fw, sc, floor, budget, s)
        torch.cuda.synchronize()
        assert st == 0, st
        for key in ("counts", "offsets", "kept_pos", "tau"):
            np.testing.assert_array_equal(np_(got[key]), np_(ref[key]), err_msg=key)
        one = np.ones(sc.shape[0])
        assert_close(np_(got["dropped_alloc"]), np_(ref["dropped_alloc"]), one, "dropped_alloc")
        assert_close(np_(got["dropped_uniform"]), np_(ref["dropped_uniform"]), one, "dropped_uniform")


def test_noalloc_at_its_largest_size_allocates_nothing(fw):
    # exactly FW_CONTOUR_NOALLOC_MAX_CELLS cells (the shared array filled to its
    # limit), bit for bit against the workspace entry point; the device's free
    # memory is the same before and after the call
    cells = 4096
    cb = workloads.contour_cache(seed=77, cells=cells, T=96, with_kv=False, budget_frac=1 / 2)
    sc = torch.as_tensor(cb.scores).cuda()
    ref = fw.contour_alloc(sc, floor=cb.floor, total_budget=cb.total_budget, uniform_s=cb.uniform_s)
    st, _ = call_noalloc(fw, sc, cb.floor, cb.total_budget, cb.uniform_s)  # the module is loaded after this
    assert st == 0, st
    got = new_outputs(cells, cb.total_budget, sc.device)  # outputs allocated before the measured call
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    st, got = call_noalloc(fw, sc, cb.floor, cb.total_budget, cb.uniform_s, out=got)
    torch.cuda.synchronize()
    free1 = torch.cuda.mem_get_info()[0]
    assert st == 0, st
    assert free1 == free0
    for key in ("counts", "offsets", "kept_pos", "tau"):
        np.testing.assert_array_equal(np_(got[key]), np_(ref[key]), err_msg=key)
    one = np.ones(cells)
    assert_close(np_(got["dropped_alloc"]), np_(ref["dropped_alloc"]), one, "dropped_alloc")
    assert_close(np_(got["dropped_uniform"]), np_(ref["dropped_uniform"]), one, "dropped_uniform")


def test_noalloc_rejects_more_cells_than_its_scratch_holds(fw):
    before = fw.launch_count()
    cells = 4097
    sc = torch.ones(cells, 64, device="cuda")
    st, _ = call_noalloc(fw, sc, 32, cells * 32, 32)
    assert st == fw.FW_ERR_WORKSPACE
    assert fw.launch_count() == before
